// Token-layout builder: summary-token insertion, position ids, window and ring
// offsets, compaction gather list (Sec. 3.2 "Setup and tokens"; App. A).
//
// Two launches. (1) One CTA scans the window lengths into each window's first
// base (fixed W, or a per-window schedule for adaptive windowing), then the
// augmented sizes T_w = n_w + B_w and kept-row counts B_w + min(tail, n_w) into
// win_off / ring_off. (2) One thread
// per augmented row locates its window by binary search over win_off and
// classifies the row in closed form: inside a window, k-mer c occupies rows
// [c(k+1), c(k+1)+len_c] with its summary at offset len_c, where
// len_c = min(k, n_w - c k). A kept row's place in the ring is the window's ring
// offset plus the summaries and boundary-tail bases before it.
#include "common.cuh"

namespace focus {
namespace {

constexpr int kScanThreads = 1024;

__device__ __forceinline__ int64_t warp_incl_scan(int64_t v) {
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        int64_t n = __shfl_up_sync(0xffffffffu, v, off);
        if ((threadIdx.x & 31) >= off) v += n;
    }
    return v;
}

// Block-wide exclusive scan of K counters; block totals via tot[].
template <int K>
__device__ void block_excl_scan(const int64_t* x, int64_t* ex, int64_t* tot) {
    __shared__ int64_t ws[K][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int64_t in[K];
#pragma unroll
    for (int c = 0; c < K; ++c) {
        in[c] = warp_incl_scan(x[c]);
        if (lane == 31) ws[c][warp] = in[c];
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int c = 0; c < K; ++c) {
            int64_t v = lane < nw ? ws[c][lane] : 0;
            v = warp_incl_scan(v);
            if (lane < nw) ws[c][lane] = v;
        }
    }
    __syncthreads();
#pragma unroll
    for (int c = 0; c < K; ++c) {
        ex[c] = (warp ? ws[c][warp - 1] : 0) + in[c] - x[c];
        tot[c] = ws[c][nw - 1];
    }
    __syncthreads();
}

// Window sizes: a first scan of the window lengths gives each window's first
// base S_w (hence n_w = min(W_w, N - S_w)), a second the augmented rows T_w and
// kept rows; the offsets are their running sums.
__global__ void __launch_bounds__(kScanThreads) layout_windows_kernel(
        int64_t N, int32_t W, const int32_t* __restrict__ Ws, int32_t M, const int32_t* __restrict__ ks,
        bool close_tail, int32_t tail, int32_t* __restrict__ win_off, int32_t* __restrict__ ring_off,
        int32_t* __restrict__ base_off, int64_t expect_T, int64_t expect_R, int32_t* status) {
    int64_t carry_S = 0, carry_T = 0, carry_R = 0;
    bool bad = false;
    for (int32_t base = 0; base < M; base += kScanThreads) {
        const int32_t w = base + (int32_t)threadIdx.x;
        int64_t len[1] = {0}, S[1], totS[1];
        if (w < M) {
            len[0] = Ws ? Ws[w] : W;
            if (len[0] <= 0) bad = true;
        }
        block_excl_scan<1>(len, S, totS);
        int64_t x[2] = {0, 0}, ex[2], tot[2];
        if (w < M) {
            const int64_t Sw = carry_S + S[0];
            if (Sw >= N) bad = true;                       // an empty window
            int64_t n = N - Sw;
            if (n > len[0]) n = len[0];
            if (n < 0) n = 0;
            const int32_t k = ks[w];
            if (k < 0) bad = true;
            const bool close = (w < M - 1) || close_tail;
            const int64_t rows = window_rows(n, k, close);
            x[0] = rows;
            x[1] = rows - n + (n - tail_start(n, tail));
            if (base_off) base_off[w] = (int32_t)Sw;
        }
        block_excl_scan<2>(x, ex, tot);
        if (w < M) {
            win_off[w] = (int32_t)(carry_T + ex[0]);
            ring_off[w] = (int32_t)(carry_R + ex[1]);
        }
        carry_S += totS[0];
        carry_T += tot[0];
        carry_R += tot[1];
    }
    if (threadIdx.x == 0) {
        win_off[M] = (int32_t)carry_T;
        ring_off[M] = (int32_t)carry_R;
        if (base_off) base_off[M] = (int32_t)N;
        if (carry_S < N) bad = true;                       // the windows do not cover the sequence
    }
    if (bad) report(status, FOCUS_ERR_INVALID_ARG);
    if (threadIdx.x == 0 && (carry_T != expect_T || carry_R != expect_R)) report(status, FOCUS_ERR_LAYOUT);
}

__global__ void __launch_bounds__(256) layout_rows_kernel(
        int64_t N, int32_t W, const int32_t* __restrict__ Ws, int32_t M, const int32_t* __restrict__ ks,
        bool close_tail, int32_t tail, int32_t B, const uint8_t* __restrict__ nt, int64_t T,
        const int32_t* __restrict__ win_off, const int32_t* __restrict__ ring_off,
        const int32_t* __restrict__ base_off, uint8_t* __restrict__ kind, int32_t* __restrict__ src,
        int32_t* __restrict__ pos, int32_t* __restrict__ win, uint8_t* __restrict__ tok,
        uint8_t* __restrict__ keep, int32_t* __restrict__ sum_idx, int64_t R) {
    int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= T) return;
    if ((int64_t)win_off[M] != T || (int64_t)ring_off[M] != R) return;  // flagged by the scan
    // largest w with win_off[w] <= t
    int32_t lo = 0, hi = M - 1;
    while (lo < hi) {
        int32_t mid = (lo + hi + 1) >> 1;
        if ((int64_t)win_off[mid] <= t) lo = mid; else hi = mid - 1;
    }
    const int32_t w = lo;
    const int64_t a = t - win_off[w];
    const int64_t S = base_off ? (int64_t)base_off[w] : (int64_t)w * W;   // first base of the window
    int64_t n = N - S;
    const int64_t len = Ws ? Ws[w] : W;
    if (n > len) n = len;
    const int32_t k = ks[w];
    const int64_t ts = tail_start(n, tail);
    int64_t s;
    bool summary = false, kept;
    int64_t ring_pos;                 // index in the ring if kept
    if (k <= 0) {
        s = S + a;
        kept = a >= ts;
        ring_pos = a - ts;
    } else {
        int64_t c = a / (k + 1), r = a % (k + 1);
        int64_t klen = n - c * k;
        if (klen > k) klen = k;
        if (r < klen) {               // base number c*k + r of the window
            const int64_t o = c * k + r;
            s = S + o;
            kept = o >= ts;
            ring_pos = c + (o - ts);  // c summaries and (o - ts) tail bases precede it
        } else {                      // summary of k-mer c, after base c*k + klen - 1
            summary = true;
            kept = true;
            s = S + c * k + klen - 1;
            const int64_t tb = c * k + klen - ts;
            ring_pos = c + (tb > 0 ? tb : 0);
        }
    }
    if (kept) sum_idx[ring_off[w] + ring_pos] = (int32_t)t;
    if (keep) keep[t] = kept ? 1 : 0;
    kind[t] = summary ? 1 : 0;
    src[t] = (int32_t)s;
    pos[t] = (int32_t)t;
    win[t] = w;
    if (tok && nt) {
        for (int32_t b = 0; b < B; ++b)
            tok[(int64_t)b * T + t] = summary ? (uint8_t)FOCUS_SUMMARY_TOKEN : nt[(int64_t)b * N + s];
    }
}

}  // namespace

cudaError_t launch_layout(int64_t N, int32_t W, const int32_t* d_W, int32_t M, const int32_t* d_k, bool close_tail,
                          int32_t tail, int32_t B, const uint8_t* d_nt, const focus_layout_out& out,
                          int32_t* status, cudaStream_t stream) {
    layout_windows_kernel<<<1, kScanThreads, 0, stream>>>(N, W, d_W, M, d_k, close_tail, tail, out.win_off,
                                                          out.ring_off, out.base_off, out.T, out.R, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || out.T == 0) return e;
    unsigned blocks = (unsigned)ceil_div64(out.T, 256);
    layout_rows_kernel<<<blocks, 256, 0, stream>>>(N, W, d_W, M, d_k, close_tail, tail, B, d_nt, out.T,
                                                   out.win_off, out.ring_off, d_W ? out.base_off : nullptr,
                                                   out.kind, out.src, out.pos, out.win, out.tok, out.keep,
                                                   out.sum_idx, out.R);
    return cudaGetLastError();
}

}  // namespace focus
