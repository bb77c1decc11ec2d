// Token-layout builder: summary-token insertion, position ids, window and ring
// offsets, compaction gather list (Sec. 3.2 "Setup and tokens"; App. A).
//
// Two launches. (1) One CTA scans the per-window augmented sizes T_w = n_w + B_w
// and kept-row counts B_w + min(tail, n_w) into win_off / ring_off. (2) One thread
// per augmented row locates its window by binary search over win_off and
// classifies the row in closed form: inside a window, k-mer c occupies rows
// [c(k+1), c(k+1)+len_c] with its summary at offset len_c, where
// len_c = min(k, n_w - c k). A kept row's place in the ring is the window's ring
// offset plus the summaries and boundary-tail bases before it.
#include "common.cuh"

namespace focus {
namespace {

constexpr int kScanThreads = 1024;

__device__ __forceinline__ int32_t warp_incl_scan(int32_t v) {
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        int32_t n = __shfl_up_sync(0xffffffffu, v, off);
        if ((threadIdx.x & 31) >= off) v += n;
    }
    return v;
}

// Block-wide exclusive scan of two counters; returns block totals via *tot.
__device__ void block_excl_scan2(int32_t a, int32_t b, int32_t* ea, int32_t* eb, int32_t* ta, int32_t* tb) {
    __shared__ int32_t wa[32], wb[32];
    int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t ia = warp_incl_scan(a), ib = warp_incl_scan(b);
    if (lane == 31) { wa[warp] = ia; wb[warp] = ib; }
    __syncthreads();
    if (warp == 0) {
        int nw = blockDim.x >> 5;
        int32_t xa = lane < nw ? wa[lane] : 0, xb = lane < nw ? wb[lane] : 0;
        xa = warp_incl_scan(xa);
        xb = warp_incl_scan(xb);
        if (lane < nw) { wa[lane] = xa; wb[lane] = xb; }
    }
    __syncthreads();
    int32_t pa = warp ? wa[warp - 1] : 0, pb = warp ? wb[warp - 1] : 0;
    *ea = pa + ia - a;
    *eb = pb + ib - b;
    *ta = wa[(blockDim.x >> 5) - 1];
    *tb = wb[(blockDim.x >> 5) - 1];
    __syncthreads();
}

__global__ void __launch_bounds__(kScanThreads) layout_windows_kernel(
        int64_t N, int32_t W, int32_t M, const int32_t* __restrict__ ks, bool close_tail, int32_t tail,
        int32_t* __restrict__ win_off, int32_t* __restrict__ ring_off, int64_t expect_T,
        int64_t expect_R, int32_t* status) {
    int32_t carry_T = 0, carry_R = 0;
    bool bad = false;
    for (int32_t base = 0; base < M; base += kScanThreads) {
        int32_t w = base + (int32_t)threadIdx.x;
        int32_t tw = 0, bw = 0;
        if (w < M) {
            int64_t n = N - (int64_t)w * W;
            if (n > W) n = W;
            int32_t k = ks[w];
            if (k < 0) bad = true;
            bool close = (w < M - 1) || close_tail;
            int64_t rows = window_rows(n, k, close);
            tw = (int32_t)rows;
            bw = (int32_t)(rows - n + (n - tail_start(n, tail)));
        }
        int32_t et, eb, tt, tb;
        block_excl_scan2(tw, bw, &et, &eb, &tt, &tb);
        if (w < M) {
            win_off[w] = carry_T + et;
            ring_off[w] = carry_R + eb;
        }
        carry_T += tt;
        carry_R += tb;
    }
    if (threadIdx.x == 0) {
        win_off[M] = carry_T;
        ring_off[M] = carry_R;
    }
    if (bad) report(status, FOCUS_ERR_INVALID_ARG);
    if (threadIdx.x == 0 && ((int64_t)carry_T != expect_T || (int64_t)carry_R != expect_R))
        report(status, FOCUS_ERR_LAYOUT);
}

__global__ void __launch_bounds__(256) layout_rows_kernel(
        int64_t N, int32_t W, int32_t M, const int32_t* __restrict__ ks, bool close_tail, int32_t tail, int32_t B,
        const uint8_t* __restrict__ nt, int64_t T, const int32_t* __restrict__ win_off,
        const int32_t* __restrict__ ring_off, uint8_t* __restrict__ kind, int32_t* __restrict__ src,
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
    int64_t n = N - (int64_t)w * W;
    if (n > W) n = W;
    const int32_t k = ks[w];
    const int64_t ts = tail_start(n, tail);
    int64_t s;
    bool summary = false, kept;
    int64_t ring_pos;                 // index in the ring if kept
    if (k <= 0) {
        s = (int64_t)w * W + a;
        kept = a >= ts;
        ring_pos = a - ts;
    } else {
        int64_t c = a / (k + 1), r = a % (k + 1);
        int64_t len = n - c * k;
        if (len > k) len = k;
        if (r < len) {                // base number c*k + r of the window
            const int64_t o = c * k + r;
            s = (int64_t)w * W + o;
            kept = o >= ts;
            ring_pos = c + (o - ts);  // c summaries and (o - ts) tail bases precede it
        } else {                      // summary of k-mer c, after base c*k + len - 1
            summary = true;
            kept = true;
            s = (int64_t)w * W + c * k + len - 1;
            const int64_t tb = c * k + len - ts;
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

cudaError_t launch_layout(int64_t N, int32_t W, int32_t M, const int32_t* d_k, bool close_tail,
                          int32_t tail, int32_t B, const uint8_t* d_nt, const focus_layout_out& out,
                          int32_t* status, cudaStream_t stream) {
    layout_windows_kernel<<<1, kScanThreads, 0, stream>>>(N, W, M, d_k, close_tail, tail, out.win_off,
                                                          out.ring_off, out.T, out.R, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || out.T == 0) return e;
    unsigned blocks = (unsigned)ceil_div64(out.T, 256);
    layout_rows_kernel<<<blocks, 256, 0, stream>>>(N, W, M, d_k, close_tail, tail, B, d_nt, out.T,
                                                   out.win_off, out.ring_off, out.kind, out.src,
                                                   out.pos, out.win, out.tok, out.keep, out.sum_idx, out.R);
    return cudaGetLastError();
}

}  // namespace focus
