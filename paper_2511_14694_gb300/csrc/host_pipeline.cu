// focus_prefill_host (include/focus.h): the masked-parallel prefill of App. A.1
// (bulk compaction of every window's FOCUS rows, then one attention call over all
// windows) for a layer whose inputs and outputs are in host memory. Host code
// only: the library's own layout, compaction and prefill calls per part of the
// heads (one sequence) or of the sequences, with the part's host<->device copies
// on two caller streams, so that the copies of one part overlap the kernels and
// copies of the others.
#include <vector>

#include "common.cuh"

namespace {

// Events this call creates; released when the call returns (the driver keeps an
// event that is still pending until the device has passed it).
struct Events {
    std::vector<cudaEvent_t> ev;
    ~Events() {
        for (cudaEvent_t e : ev) cudaEventDestroy(e);
    }
    // `waiter` waits for everything enqueued on `s` so far
    cudaError_t order(cudaStream_t waiter, cudaStream_t s) {
        cudaEvent_t e;
        cudaError_t r = cudaEventCreateWithFlags(&e, cudaEventDisableTiming);
        if (r != cudaSuccess) return r;
        ev.push_back(e);
        if ((r = cudaEventRecord(e, s)) != cudaSuccess) return r;
        return cudaStreamWaitEvent(waiter, e, 0);
    }
};

// p advanced by elems elements of elem_bytes each (NULL stays NULL)
template <typename P>
P offset(P p, size_t elems, size_t elem_bytes) {
    return p ? (P)((const char*)p + elems * elem_bytes) : p;
}

}  // namespace

extern "C" focus_status focus_prefill_host(const focus_cache* cache, const focus_prefill_host_args* a,
                                           cudaStream_t stream) {
    if (!cache || !a || !a->layout) return FOCUS_ERR_INVALID_ARG;
    if (!a->h_nt || !a->h_q || !a->h_k || !a->h_v || !a->h_o || !a->d_nt || !a->d_q || !a->d_k || !a->d_v ||
        !a->d_o || (a->h_lse && !a->d_lse))
        return FOCUS_ERR_INVALID_ARG;
    if (a->groups < 1 || a->copy_in == stream || a->copy_out == stream || a->copy_in == a->copy_out)
        return FOCUS_ERR_INVALID_ARG;
    if (cache->B <= 0 || cache->H <= 0 || (cache->d != 64 && cache->d != 128) || a->n_nt < 0 || a->n_windows < 0)
        return FOCUS_ERR_INVALID_ARG;
    const focus_cache& c = *cache;
    const focus_layout_out& L = *a->layout;
    const size_t B = (size_t)c.B, H = (size_t)c.H, d = (size_t)c.d, T = (size_t)L.T;
    const size_t g = c.q_per_kv > 1 ? (size_t)c.q_per_kv : 1;
    Events E;
#define FOCUS_CU(x)                                       \
    do {                                                  \
        if ((x) != cudaSuccess) return FOCUS_ERR_CUDA;    \
    } while (0)
    // the previous call's kernels and copies out are done with the device buffers
    FOCUS_CU(E.order(a->copy_in, stream));
    FOCUS_CU(E.order(a->copy_in, a->copy_out));
    FOCUS_CU(cudaMemcpyAsync(a->d_nt, a->h_nt, B * (size_t)a->n_nt, cudaMemcpyHostToDevice, a->copy_in));
    FOCUS_CU(E.order(stream, a->copy_in));
    focus_status s = a->d_W_sched
                         ? focus_layout_sched(a->n_nt, a->n_windows, a->d_W_sched, a->d_k_sched, a->layout_flags,
                                              a->tail, c.B, a->d_nt, a->layout, stream)
                         : focus_layout(a->n_nt, a->W, a->n_windows, a->d_k_sched, a->layout_flags, a->tail, c.B,
                                        a->d_nt, a->layout, stream);
    if (s != FOCUS_OK) return s;
    if (T == 0) return FOCUS_OK;
    // parts: K/V heads of the one sequence, or sequences; each is contiguous in
    // every tensor (q heads of K/V head h are h g .. h g + g - 1)
    const bool by_head = B == 1;
    const size_t n = by_head ? H : B;
    const size_t groups = (size_t)a->groups < n ? (size_t)a->groups : n;
    const size_t kv_unit = by_head ? T * d : H * T * d;        // elements of one part unit in k, v
    const size_t q_unit = kv_unit * g;                          // ... in q, o
    const size_t lse_unit = (by_head ? T : H * T) * g;          // ... in lse
    for (size_t i = 0; i < groups; ++i) {
        const size_t lo = n * i / groups, hi = n * (i + 1) / groups, m = hi - lo;
        if (m == 0) continue;
        FOCUS_CU(cudaMemcpyAsync(offset(a->d_q, lo * q_unit, 2), offset(a->h_q, lo * q_unit, 2), m * q_unit * 2,
                                 cudaMemcpyHostToDevice, a->copy_in));
        FOCUS_CU(cudaMemcpyAsync(offset(a->d_k, lo * kv_unit, 2), offset(a->h_k, lo * kv_unit, 2), m * kv_unit * 2,
                                 cudaMemcpyHostToDevice, a->copy_in));
        FOCUS_CU(cudaMemcpyAsync(offset(a->d_v, lo * kv_unit, 2), offset(a->h_v, lo * kv_unit, 2), m * kv_unit * 2,
                                 cudaMemcpyHostToDevice, a->copy_in));
        FOCUS_CU(E.order(stream, a->copy_in));
        // the part's view of the cache
        focus_cache p = c;
        const size_t ring_unit = (by_head ? 1 : H) * (size_t)c.C_ring * d, win_unit = (by_head ? 1 : H) * (size_t)c.C_win * d;
        p.ring_k = offset(c.ring_k, lo * ring_unit, 2);
        p.ring_v = offset(c.ring_v, lo * ring_unit, 2);
        p.win_k = offset(c.win_k, lo * win_unit, 2);
        p.win_v = offset(c.win_v, lo * win_unit, 2);
        if (by_head) {
            p.H = (int32_t)m;
        } else {
            p.B = (int32_t)m;
            p.ring_len = offset(c.ring_len, lo, 4);
            p.win_fill = offset(c.win_fill, lo, 4);
            p.win_idx = offset(c.win_idx, lo, 4);
            p.pos_base = offset(c.pos_base, lo, 4);
        }
        focus_compact_args ca = {};
        ca.src_k = offset(a->d_k, lo * kv_unit, 2);
        ca.src_v = offset(a->d_v, lo * kv_unit, 2);
        ca.src_T = (int64_t)T;
        ca.src_row0 = 0;
        ca.d_sum_idx = L.sum_idx;
        ca.d_ring_off = L.ring_off;
        ca.n_windows = a->n_windows;
        ca.w_begin = 0;
        ca.w_end = a->n_windows;
        if ((s = focus_kv_compact(&p, &ca, stream)) != FOCUS_OK) return s;
        focus_prefill_args pa = {};
        pa.q = offset(a->d_q, lo * q_unit, 2);
        pa.k = ca.src_k;
        pa.v = ca.src_v;
        pa.o = offset(a->d_o, lo * q_unit, 2);
        pa.lse = a->h_lse ? offset(a->d_lse, lo * lse_unit, 4) : nullptr;
        pa.T_span = (int64_t)T;
        pa.d_win_off = L.win_off;
        pa.d_ring_off = L.ring_off;
        pa.n_windows = a->n_windows;
        pa.w_begin = 0;
        pa.w_end = a->n_windows;
        pa.max_rows = a->max_rows;
        pa.scale = a->scale;
        pa.flags = a->prefill_flags;
        pa.workspace = a->workspace;
        pa.workspace_bytes = a->workspace_bytes;
        if ((s = focus_attn_prefill(&p, &pa, stream)) != FOCUS_OK) return s;
        FOCUS_CU(E.order(a->copy_out, stream));
        FOCUS_CU(cudaMemcpyAsync(offset(a->h_o, lo * q_unit, 2), pa.o, m * q_unit * 2, cudaMemcpyDeviceToHost,
                                 a->copy_out));
        if (a->h_lse)
            FOCUS_CU(cudaMemcpyAsync(offset(a->h_lse, lo * lse_unit, 4), pa.lse, m * lse_unit * 4,
                                     cudaMemcpyDeviceToHost, a->copy_out));
    }
    FOCUS_CU(E.order(stream, a->copy_out));
#undef FOCUS_CU
    return FOCUS_OK;
}
