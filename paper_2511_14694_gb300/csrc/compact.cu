// KV retention / compaction (App. A, "KV compression and budget"; Sec. 3.2
// "KV retention and memory profile"): after a window, only the FOCUS rows' K/V
// (and, if asked for, the window's boundary tail of ordinary rows) are kept,
// appended to the per-(sequence, head) ring. Other rows are simply not copied.
// Pure data movement, bit-exact; 16-byte vector loads and stores.
#include "common.cuh"
#include "sm100.cuh"

namespace focus {
namespace {

// Bulk mode: ring[b,h, r] <- src[b,h, sum_idx[r] - src_row0] for r in
// [ring_off[w_begin], ring_off[w_end]). One warp per unit of 64 ring rows of one
// (sequence, head): its lanes gather the rows' K and V into shared memory with
// one cp.async.bulk per row (the copy engine keeps far more bytes in flight than
// per-thread loads, whose outstanding misses per SM are capped), and since the
// unit's ring rows are contiguous, two bulk stores write it out.
constexpr int kBulkRows = 64;

template <int D>
__global__ void __launch_bounds__(32) compact_bulk_kernel(
        uint8_t* __restrict__ ring_k, uint8_t* __restrict__ ring_v, const uint8_t* __restrict__ src_k,
        const uint8_t* __restrict__ src_v, int32_t BH, int32_t B, int32_t C_ring, int64_t src_T, int64_t src_row0,
        const int32_t* __restrict__ sum_idx, const int32_t* __restrict__ ring_off, int32_t w_begin, int32_t w_end,
        int32_t* __restrict__ ring_len, int32_t* status) {
    using namespace sm100;
    constexpr int ROWB = 2 * D;
    __shared__ __align__(128) uint8_t sk[kBulkRows * ROWB];
    __shared__ __align__(128) uint8_t sv[kBulkRows * ROWB];
    __shared__ uint64_t bar;
    const int lane = threadIdx.x;
    const int32_t r0 = ring_off[w_begin], r1 = ring_off[w_end];
    if (r1 > C_ring) {
        if (blockIdx.x == 0 && lane == 0) report(status, FOCUS_ERR_CAPACITY);
        return;
    }
    if (lane == 0) {
        mbar_init(smem_addr(&bar), 1);
        fence_barrier_init();
    }
    __syncwarp();
    const int32_t nrb = (r1 - r0 + kBulkRows - 1) / kBulkRows;
    const int64_t units = (int64_t)nrb * BH;
    uint32_t phase = 0;
    for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
        const int32_t rs = r0 + (int32_t)(u % nrb) * kBulkRows;
        const int64_t bh = u / nrb;
        const int32_t rows = r1 - rs < kBulkRows ? r1 - rs : kBulkRows;
        // each lane owns rows lane and lane + 32 of the unit
        int64_t srow[2];
        bool bad = false;
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int i = lane + 32 * q;
            srow[q] = i < rows ? (int64_t)sum_idx[rs + i] - src_row0 : 0;
            if (i < rows && (srow[q] < 0 || srow[q] >= src_T)) bad = true;
        }
        if (__any_sync(0xffffffffu, bad)) {
            if (lane == 0) report(status, FOCUS_ERR_INVALID_ARG);
            continue;
        }
        if (lane == 0) mbar_expect_tx(smem_addr(&bar), (uint32_t)(rows * 2 * ROWB));
        __syncwarp();
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int i = lane + 32 * q;
            if (i < rows) {
                const int64_t so = (bh * src_T + srow[q]) * ROWB;
                bulk_load(smem_addr(sk + i * ROWB), src_k + so, ROWB, smem_addr(&bar));
                bulk_load(smem_addr(sv + i * ROWB), src_v + so, ROWB, smem_addr(&bar));
            }
        }
        if (!mbar_wait(smem_addr(&bar), phase, 2000000000ull)) {
            if (lane == 0) report(status, FOCUS_ERR_TIMEOUT);
            break;
        }
        phase ^= 1u;
        if (lane == 0) {
            const int64_t d_o = (bh * C_ring + rs) * ROWB;
            bulk_store(ring_k + d_o, smem_addr(sk), (uint32_t)(rows * ROWB));
            bulk_store(ring_v + d_o, smem_addr(sv), (uint32_t)(rows * ROWB));
            bulk_commit();
            bulk_wait_read_all();              // the buffers are reused by the next unit
        }
        __syncwarp();
    }
    if (lane == 0) bulk_wait_all();            // the ring rows are written before the CTA exits
    if (blockIdx.x == 0)
        for (int32_t b = lane; b < B; b += 32) ring_len[b] = r1;
}

// Bulk mode with the rotary embedding: ring K rows are stored rotated at their
// position id p = sum_idx[r]. One thread owns one ring row, one pair of 16-byte
// chunks (columns 8j.. and 8j + d/2..) and a group of four (sequence, head)
// pairs: it forms the eight angles p theta_i (fp64 product, reduced) and applies
// them to each pair of the group; V is copied as is.
template <int D>
__global__ void __launch_bounds__(256) compact_bulk_rope_kernel(
        uint4* __restrict__ ring_k, uint4* __restrict__ ring_v, const uint4* __restrict__ src_k,
        const uint4* __restrict__ src_v, int32_t BH, int32_t B, int32_t C_ring, int64_t src_T, int64_t src_row0,
        const int32_t* __restrict__ sum_idx, const int32_t* __restrict__ ring_off, int32_t w_begin, int32_t w_end,
        int32_t* __restrict__ ring_len, const __grid_constant__ RopeTable rope, int32_t* status) {
    constexpr int CPR = D / 8, HALF = D / 16;   // chunks per row, chunk pairs per row
    const int32_t r0 = ring_off[w_begin], r1 = ring_off[w_end];
    const int64_t rows = r1 - r0;
    if (r1 > C_ring) {
        if (blockIdx.x == 0 && threadIdx.x == 0) report(status, FOCUS_ERR_CAPACITY);
        return;
    }
    // work unit: (group of U (sequence, head) pairs, ring row, chunk pair), the
    // group outermost, so that a warp covers whole ring rows of one group and the
    // launch has rows x d/16 x ceil(BH / U) threads' worth of units
    constexpr int U = 4;
    const int64_t units = rows * HALF, n_groups = (BH + U - 1) / U;
    for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < units * n_groups;
         x += (int64_t)gridDim.x * blockDim.x) {
        const int64_t grp = x / units, u = x - grp * units;
        const int j = (int)(u % HALF);
        const int64_t r = r0 + u / HALF;
        const int64_t p = sum_idx[r];
        const int64_t srow = p - src_row0;
        if (srow < 0 || srow >= src_T) {
            report(status, FOCUS_ERR_INVALID_ARG);
            continue;
        }
        float2 cs[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) cs[e] = rope_cs((double)p * rope.theta[8 * j + e]);
        const int64_t bh0 = grp * U;
        if (bh0 + U <= BH) {                     // U rows' loads in flight
            uint4 klo[U], khi[U], vlo[U], vhi[U];
#pragma unroll
            for (int e = 0; e < U; ++e) {
                const int64_t so = ((bh0 + e) * src_T + srow) * CPR;
                klo[e] = src_k[so + j];
                khi[e] = src_k[so + j + HALF];
                vlo[e] = src_v[so + j];
                vhi[e] = src_v[so + j + HALF];
            }
#pragma unroll
            for (int e = 0; e < U; ++e) {
                const int64_t d_o = ((bh0 + e) * C_ring + r) * CPR;
                rope_rotate8(klo[e], khi[e], cs);
                ring_k[d_o + j] = klo[e];
                ring_k[d_o + j + HALF] = khi[e];
                ring_v[d_o + j] = vlo[e];
                ring_v[d_o + j + HALF] = vhi[e];
            }
        } else {
            for (int64_t bh = bh0; bh < BH; ++bh) {
                const int64_t so = (bh * src_T + srow) * CPR, d_o = (bh * C_ring + r) * CPR;
                uint4 lo = src_k[so + j], hi = src_k[so + j + HALF];
                rope_rotate8(lo, hi, cs);
                ring_k[d_o + j] = lo;
                ring_k[d_o + j + HALF] = hi;
                ring_v[d_o + j] = src_v[so + j];
                ring_v[d_o + j + HALF] = src_v[so + j + HALF];
            }
        }
    }
    if (blockIdx.x == 0)
        for (int32_t b = threadIdx.x; b < B; b += blockDim.x) ring_len[b] = r1;
}

// Window mode: one CTA per sequence. If the current window buffer holds the
// whole window (W bases + its summaries), append its kept rows (FOCUS rows and
// the last `tail` bases) to the ring in augmented order and start the next
// window. Kept row j is either summary j (j < B_w) or tail base j - B_w; each
// one's buffer row and ring slot follow in closed form.
__global__ void __launch_bounds__(256) compact_window_kernel(
        uint4* __restrict__ ring_k, uint4* __restrict__ ring_v, const uint4* __restrict__ win_k,
        const uint4* __restrict__ win_v, int32_t* __restrict__ ring_len, int32_t* __restrict__ win_fill,
        int32_t* __restrict__ win_idx, const int32_t* __restrict__ ks, int32_t n_windows, int32_t W_fixed,
        int32_t H, int32_t chunks_per_row, int32_t C_ring, int32_t C_win, int32_t tail,
        int32_t* __restrict__ pos_base, int32_t* status, const int32_t* __restrict__ W_per_window) {
    const int32_t b = blockIdx.x;
    const int32_t fill = win_fill[b], widx = win_idx[b], R = ring_len[b];
    if (widx < 0 || widx >= n_windows) {
        if (threadIdx.x == 0) report(status, FOCUS_ERR_CAPACITY);
        return;
    }
    const int32_t k = ks[widx];
    const int32_t W = cache_window_len(W_per_window, W_fixed, widx);
    const int32_t Tw = (int32_t)window_rows(W, k, true);
    if (fill != Tw) return;                  // window not complete yet
    const int32_t Bw = Tw - W;
    const int32_t ts = (int32_t)tail_start(W, tail);
    const int32_t kept = Bw + (W - ts);
    if (R + kept > C_ring || Tw > C_win) {
        if (threadIdx.x == 0) report(status, FOCUS_ERR_CAPACITY);
        return;
    }
    const int64_t total = (int64_t)H * kept * chunks_per_row;
    for (int64_t i = threadIdx.x; i < total; i += blockDim.x) {
        const int32_t c = (int32_t)(i % chunks_per_row);
        const int64_t rest = i / chunks_per_row;
        const int32_t j = (int32_t)(rest % kept);
        const int64_t h = rest / kept;
        const int64_t bh = (int64_t)b * H + h;
        int32_t row, slot;
        if (j < Bw) {                       // summary j, after base min((j+1)k, W) - 1
            row = window_summary_row(j, W, k);
            const int32_t end = (int64_t)(j + 1) * k < W ? (j + 1) * k : W;
            slot = j + (end > ts ? end - ts : 0);
        } else {                            // tail base o
            const int32_t o = ts + (j - Bw);
            const int32_t before = k > 0 ? o / k : 0;   // summaries before base o
            row = o + before;
            slot = before + (j - Bw);
        }
        const int64_t so = (bh * C_win + row) * chunks_per_row + c;
        const int64_t d_o = (bh * C_ring + R + slot) * chunks_per_row + c;
        ring_k[d_o] = win_k[so];
        ring_v[d_o] = win_v[so];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        ring_len[b] = R + kept;
        win_fill[b] = 0;
        win_idx[b] = widx + 1;
        if (pos_base) pos_base[b] += Tw;
    }
}

}  // namespace

cudaError_t launch_compact_bulk(const focus_cache& c, const focus_compact_args& a, int32_t* status,
                                cudaStream_t stream) {
    // the span's row count lives on the device (ring_off): at most one warp per
    // possible unit, at most eight per SM; each strides over the units
    int dev = 0, sms = 152;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t BH = (int64_t)c.B * c.H;
    int64_t grid = ceil_div64(c.C_ring > 0 ? c.C_ring : 1, kBulkRows) * BH;
    if (grid > 8 * (int64_t)sms) grid = 8 * (int64_t)sms;
    if (c.d == 128)
        compact_bulk_kernel<128><<<(unsigned)grid, 32, 0, stream>>>(
            (uint8_t*)c.ring_k, (uint8_t*)c.ring_v, (const uint8_t*)a.src_k, (const uint8_t*)a.src_v, (int32_t)BH,
            c.B, c.C_ring, a.src_T, a.src_row0, a.d_sum_idx, a.d_ring_off, a.w_begin, a.w_end, c.ring_len, status);
    else
        compact_bulk_kernel<64><<<(unsigned)grid, 32, 0, stream>>>(
            (uint8_t*)c.ring_k, (uint8_t*)c.ring_v, (const uint8_t*)a.src_k, (const uint8_t*)a.src_v, (int32_t)BH,
            c.B, c.C_ring, a.src_T, a.src_row0, a.d_sum_idx, a.d_ring_off, a.w_begin, a.w_end, c.ring_len, status);
    return cudaGetLastError();
}

cudaError_t launch_compact_window(const focus_cache& c, int32_t* status, cudaStream_t stream) {
    compact_window_kernel<<<c.B, 256, 0, stream>>>(
        (uint4*)c.ring_k, (uint4*)c.ring_v, (const uint4*)c.win_k, (const uint4*)c.win_v, c.ring_len,
        c.win_fill, c.win_idx, c.k_per_window, c.n_windows, c.W, c.H, c.d / 8, c.C_ring, c.C_win, c.tail,
        c.pos_base, status, c.W_per_window);
    return cudaGetLastError();
}

cudaError_t launch_compact_bulk_rope(const focus_cache& c, const focus_compact_args& a, int32_t* status,
                                     cudaStream_t stream) {
    int dev = 0, sms = 152;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    RopeTable rope;
    rope_table_fill(&rope, c.d, c.rope_theta);
    if (c.d == 128)
        compact_bulk_rope_kernel<128><<<sms * 2, 256, 0, stream>>>(
            (uint4*)c.ring_k, (uint4*)c.ring_v, (const uint4*)a.src_k, (const uint4*)a.src_v, c.B * c.H, c.B,
            c.C_ring, a.src_T, a.src_row0, a.d_sum_idx, a.d_ring_off, a.w_begin, a.w_end, c.ring_len, rope, status);
    else
        compact_bulk_rope_kernel<64><<<sms * 2, 256, 0, stream>>>(
            (uint4*)c.ring_k, (uint4*)c.ring_v, (const uint4*)a.src_k, (const uint4*)a.src_v, c.B * c.H, c.B,
            c.C_ring, a.src_T, a.src_row0, a.d_sum_idx, a.d_ring_off, a.w_begin, a.w_end, c.ring_len, rope, status);
    return cudaGetLastError();
}

}  // namespace focus
