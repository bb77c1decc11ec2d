// Persistent variant of the tcgen05 prefill kernel for short work items
// (appendix mask, no rotary embedding): one CTA per SM walks the work items in
// rounds, so that the start-up of item i+1 (its Q and first K/V loads, its first
// QK) and the epilogue of item i overlap the other item's tiles.
//
// Same computation as prefill_tc.cu (Eq. focus-attn's visible set; App.
// A.1-A.2): row a of window w attends to ring rows [0, ring_off[w]) and to window
// rows [0, a]. Same warp roles and TMEM columns; what changes is that every
// barrier phase runs on across items:
//   warp 0     TMA producer: per item, Q tiles (once the previous item's last QK
//              has completed: q_free), then one group per MMA iteration j, {V_{j-1},
//              K_j}, into one of two stages of two slots each; one mbarrier per
//              stage, whose phase counts on across items. After an item's first
//              group it forms the next item's geometry and prefetches that item's
//              Q tiles into L2, so the Q load after q_free does not wait on DRAM
//   warp 1     MMA issuer: per item as in prefill_tc.cu, but with one stage wait
//              and one stage release per iteration; an item's first PV into O_t
//              waits until the previous item's epilogue has read O_t (o_free)
//   warps 2-3  idle; with the rotary embedding (ROPE, taken for grouped-query
//              heads; otherwise rope.cu's pass rotates q and k before this kernel)
//              they rotate the span's Q and K rows once, into a caller workspace
//              that the Q/K tensor maps read (RopeSpan below), one head ahead of
//              the attention
//   warps 4-11 softmax per tile (the shared softmax_tile), then the epilogue:
//              O_t / l to bf16 through a per-warp staging buffer (the Q buffers may
//              already hold the next item's Q), arrive on o_free once O_t is read
// Register split: warpgroup 0 keeps 104 registers (the item loops carry more state
// than the one-item kernel's 56 allow without spills), the softmax warpgroups take
// 200: 128 x 104 + 256 x 200 = 384 x 168.
// The tensor core queues about one MMA ahead of its issuing thread, so every
// instruction the issuer runs between MMA blocks (a satisfied mbarrier wait
// costs ~100 cycles) leaves the pipe idle: hence the grouped stages (one wait
// instead of two per iteration) and descriptors formed once per tile (issue_qk,
// issue_pv).
// Every mbarrier wait is bounded; on timeout the kernel reports
// FOCUS_ERR_TIMEOUT, drains its own copies/MMAs (bounded), frees TMEM, returns.
#include "prefill_tc_common.cuh"

namespace focus {
namespace prefill {
namespace {

// Register split: warpgroup 0 (TMA, MMA and, with the rotary embedding, the
// rotating warps 2-3) and the two softmax warpgroups; the counts sum to the
// launch's 384 x 168.
template <bool ROPE>
constexpr int kRegsIssue = ROPE ? 136 : 104;
template <bool ROPE>
constexpr int kRegsSoftmax = ROPE ? 184 : 200;
static_assert(128 * kRegsIssue<false> + 256 * kRegsSoftmax<false> <= kThreads * kLaunchRegs, "register split over budget");
static_assert(128 * kRegsIssue<true> + 256 * kRegsSoftmax<true> <= kThreads * kLaunchRegs, "register split over budget");

// Geometry of one work item: two 128-row Q tiles of one (sequence, head,
// window). Items are numbered head by head (sequences, then K/V heads, outermost;
// within a head the windows longest first, each window's Q-tile pairs longest
// first, and with GQA the query heads of a group innermost): the CTAs working
// at the same time then share one head's K/V tiles in L2.
struct ItemGeom {
    int32_t w, cta, member, bh, Tw, a0, Rw, row_base;
    int32_t n_ring, n_kv0, n_kv1, n_kv_max;
    bool valid, cap_err;
};

// idx < n_items < 2^31 (the host's condition for this kernel), so the index
// arithmetic is 32-bit: every role forms an item's geometry at every item.
// w0 = win_off[w_begin]; span_ok: the span's rows fit T_span (per launch).
template <bool GQA>
__device__ __forceinline__ ItemGeom item_geom(int64_t idx, uint32_t per_head, uint32_t ctas_pw, uint32_t q_per_kv,
                                              uint32_t H, const int32_t* __restrict__ win_off,
                                              const int32_t* __restrict__ ring_off, int32_t w0, bool span_ok,
                                              int32_t w_end, int32_t C_ring) {
    ItemGeom I;
    // per_head: items of one K/V head = windows x pairs (x query heads per group)
    const uint32_t u = (uint32_t)idx;
    const uint32_t rest = u / per_head, x = u - rest * per_head;
    const uint32_t b = rest / H, h = rest - b * H;
    const uint32_t item = GQA ? x / q_per_kv : x;
    I.member = GQA ? (int32_t)(x - item * q_per_kv) : 0;
    const uint32_t wi = item / ctas_pw;
    I.cta = (int32_t)(ctas_pw - 1 - (item - wi * ctas_pw));
    I.w = w_end - 1 - (int32_t)wi;
    I.bh = (int32_t)(b * H + h);
    const int32_t w_first = win_off[I.w];
    I.Tw = win_off[I.w + 1] - w_first;
    I.a0 = I.cta * 2 * BM;
    I.valid = I.a0 < I.Tw;
    I.cap_err = false;
    I.Rw = ring_off[I.w];
    I.n_ring = (I.Rw + BN - 1) / BN;
    if (I.valid && (I.Rw > C_ring || !span_ok)) {
        I.cap_err = true;
        I.valid = false;
    }
    I.row_base = w_first - w0;                          // first row of the window in the span tensors
    const bool valid1 = I.a0 + BM < I.Tw;
    I.n_kv0 = I.n_ring + 2 * I.cta + 1;
    I.n_kv1 = valid1 ? I.n_ring + 2 * I.cta + 2 : 0;
    I.n_kv_max = valid1 ? I.n_kv1 : I.n_kv0;
    return I;
}

// Rotary embedding of the span (ROPE variants). Work unit = 64 consecutive
// positions of one K/V head bh: its 64 K rows and the 64 rows of each of its g
// query heads at the same positions (one 16 KB block per row set at d = 128),
// which share every rotation angle. Units are numbered head-major (unit u: head
// u / n_chunks, rows 64 (u % n_chunks) ..), so they finish in the order the items
// use them. A group of 64 threads (tau = 0..63, its own named barrier and
// kRopeGroupScratch bytes of shared memory) takes units u0, u0 + du, ... below
// u1; after a unit, rot_done[bh] is incremented (release), and the producer
// loads a head's Q/K tiles once rot_done[bh] reaches n_chunks. Row i of the span
// has position id p_span0 + i (the span's rows are consecutive augmented rows).
//
// Thread tau owns pair chunk jj (pairs 8 jj .. 8 jj + 7: the 16-byte chunk jj and
// its partner D/2 columns on) of rows gg, gg + G, ... of each row set: the unit's
// start angle is formed per pair in fp64 and reduced modulo 2 pi (rope_cs, one
// per thread), the row offset gg theta and the stride G theta are small fp32
// angles, and the rows follow by the angle-addition recurrence.
//
// Rows move through registers only: the attention's MMAs read their operands
// from shared memory at a high rate, and staging the rows there (cp.async) made
// the rotation several times slower next to them. Each thread keeps the loads
// of kRotRows rows of two row sets in flight, and each group prefetches its next
// unit's rows into L2.
template <int D>
struct RopeSpan {
    static constexpr int HALF = D / 16, G = 64 / HALF, RPT = 64 / G, CPR = D / 8;
    static constexpr int kRotRows = 2;

    const double* theta;
    const uint4* q_src;
    const uint4* k_src;
    uint4* q_dst;
    uint4* k_dst;
    int32_t* rot_done;
    int64_t T_span;
    int32_t g;
    int32_t p_span0;
    int32_t BH;                                        // K/V heads of the span (sequences x heads)

    __device__ __forceinline__ int32_t n_chunks() const { return (int32_t)((T_span + 63) / 64); }

    // bulk prefetch into L2 of the K and Q rows of unit (bh, chunk)
    __device__ __forceinline__ void prefetch(int32_t bh, int32_t chunk) const {
        const int64_t row0 = (int64_t)chunk * 64;
        const int64_t rows = T_span - row0 < 64 ? T_span - row0 : 64;
        const uint32_t bytes = (uint32_t)(rows * D * 2);
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;"
                     ::"l"(reinterpret_cast<uint64_t>(k_src + ((int64_t)bh * T_span + row0) * CPR)), "r"(bytes)
                     : "memory");
        for (int m = 0; m < g; ++m)
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;"
                         ::"l"(reinterpret_cast<uint64_t>(q_src + (((int64_t)bh * g + m) * T_span + row0) * CPR)),
                         "r"(bytes)
                         : "memory");
    }

    // Rows gg + G m, m in [m0, m0 + kRotRows), of row sets s0 and s0 + 1 (set 0: K,
    // set 1 + i: query head i of the group) of the unit at span row row0: loads
    // first, then each row rotated by rot, which steps G positions after each.
    __device__ __forceinline__ void rows_apply(int32_t bh, int64_t row0, int gg, int m0, int rows, int s0, int jj,
                                               Rot8& rot, const Rot8& step) const {
        const bool two = s0 + 1 <= g;
        const int64_t h0 = s0 == 0 ? (int64_t)bh : (int64_t)bh * g + (s0 - 1);
        const int64_t base0 = (h0 * T_span + row0 + gg + G * m0) * CPR + jj;
        const int64_t base1 = (((int64_t)bh * g + s0) * T_span + row0 + gg + G * m0) * CPR + jj;
        const uint4* src0 = (s0 == 0 ? k_src : q_src) + base0;
        uint4* dst0 = (s0 == 0 ? k_dst : q_dst) + base0;
        uint4 lo0[kRotRows], hi0[kRotRows], lo1[kRotRows], hi1[kRotRows];
#pragma unroll
        for (int i = 0; i < kRotRows; ++i) {
            if (gg + G * (m0 + i) < rows) {
                lo0[i] = src0[i * G * CPR];
                hi0[i] = src0[i * G * CPR + HALF];
                if (two) {
                    lo1[i] = q_src[base1 + i * G * CPR];
                    hi1[i] = q_src[base1 + i * G * CPR + HALF];
                }
            }
        }
#pragma unroll
        for (int i = 0; i < kRotRows; ++i) {
            if (gg + G * (m0 + i) < rows) {
                rot8_apply(lo0[i], hi0[i], rot);
                dst0[i * G * CPR] = lo0[i];
                dst0[i * G * CPR + HALF] = hi0[i];
                if (two) {
                    rot8_apply(lo1[i], hi1[i], rot);
                    q_dst[base1 + i * G * CPR] = lo1[i];
                    q_dst[base1 + i * G * CPR + HALF] = hi1[i];
                }
            }
            rot8_step(rot, step);
        }
    }

    // scratch: kb[64] unit start angles, then 64 x 8 row offsets (float2)
    __device__ __forceinline__ void run(int32_t u0, int32_t u1, int32_t du, int tau, uint32_t bar,
                                        float2* kb) const {
        const int jj = tau % HALF, gg = tau / HALF;
        float2* off = kb + 64 + tau * 8;
        Rot8 step;
        {
            float2 o[8];
            rope_offsets(theta, 8 * jj, gg, G, o, step);
#pragma unroll
            for (int e = 0; e < 8; ++e) off[e] = o[e];
        }
        const int32_t nck = n_chunks();
        if (u1 > nck * BH) u1 = nck * BH;              // units exist for heads < BH only
        // unit u = (bh, chunk), advanced incrementally (du may exceed nck)
        int32_t bh = u0 / nck, chunk = u0 % nck;
        const int32_t dbh = du / nck, dch = du % nck;
        if (tau == 0 && u0 < u1) prefetch(bh, chunk);
        for (int32_t u = u0; u < u1; u += du) {
            int32_t nbh = bh + dbh, nch = chunk + dch;
            if (nch >= nck) {
                nch -= nck;
                ++nbh;
            }
            if (tau == 0 && u + du < u1) prefetch(nbh, nch);
            const int64_t row0 = (int64_t)chunk * 64;
            const int rows = (int)(T_span - row0 < 64 ? T_span - row0 : 64);
            if (tau < D / 2) kb[tau] = rope_cs((double)(p_span0 + row0) * theta[tau]);
            named_bar_sync(bar, 64);
            // row sets in pairs (K with the first query head, then query heads two at
            // a time), each pair's rows from the unit's start rotation
            for (int s0 = 0; s0 <= g; s0 += 2) {
                float2 cs[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) cs[e] = rope_mul(kb[8 * jj + e], off[e]);
                Rot8 rot = rot8_make(cs);
#pragma unroll 1
                for (int m0 = 0; m0 < RPT; m0 += kRotRows) rows_apply(bh, row0, gg, m0, rows, s0, jj, rot, step);
            }
            fence_proxy_async_global();
            __threadfence();
            named_bar_sync(bar, 64);                   // the unit's rows are stored; kb may be rewritten
            if (tau == 0) red_release_add(rot_done + bh, 1);
            bh = nbh;
            chunk = nch;
        }
    }
};

template <int D, bool GQA, bool ROPE>
__global__ void __launch_bounds__(kThreads, 1) prefill_tc_persistent_kernel(
        const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
        const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_rk,
        const __grid_constant__ CUtensorMap tm_rv, __nv_bfloat16* __restrict__ o, float* __restrict__ lse,
        int64_t T_span, const int32_t* __restrict__ win_off, const int32_t* __restrict__ ring_off, int32_t w_begin,
        int32_t w_end, int32_t ctas_pw, int32_t H, int32_t C_ring, float scale_log2, int32_t* status,
        int32_t q_per_kv, int64_t n_items, const __grid_constant__ RopeArg<ROPE> rope,
        const uint4* __restrict__ q_src, const uint4* __restrict__ k_src, uint4* __restrict__ q_rot,
        uint4* __restrict__ k_rot, int32_t* __restrict__ rot_done, int32_t BHk, int32_t rope_pro_heads) {
    using C = Cfg<D>;
    extern __shared__ unsigned char smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    Bars* bars = reinterpret_cast<Bars*>(smem + C::kBarOff);
    // Once any CTA has given up on a wait, CTAs that start later skip their work so
    // that a systematic stall costs one round of bounded waits.
    if (*(volatile int32_t*)status == FOCUS_ERR_TIMEOUT) return;
    const int32_t per_head = (w_end - w_begin) * ctas_pw * (GQA ? q_per_kv : 1);
    const int32_t w0 = win_off[w_begin];
    const bool span_ok = (int64_t)(win_off[w_end] - w0) <= T_span;
    auto geom = [&](int64_t idx) {
        return item_geom<GQA>(idx, (uint32_t)per_head, (uint32_t)ctas_pw, (uint32_t)q_per_kv, (uint32_t)H, win_off,
                              ring_off, w0, span_ok, w_end, C_ring);
    };
    // round k of a CTA: positions k G .. k G + G - 1 of the longest-first order, in
    // snake order (forward on even rounds, backward on odd) to balance the CTAs
    auto snake_item = [&](int64_t k) {
        return k * (int64_t)gridDim.x + ((k & 1) ? (int64_t)(gridDim.x - 1 - blockIdx.x) : (int64_t)blockIdx.x);
    };
    // the first valid item of round k or later (k is left at its round); .valid is
    // false when none is left. cap_report: report items beyond the capacities.
    auto next_valid = [&](int64_t& k, bool cap_report) {
        ItemGeom I;
        I.valid = false;
        for (; k * (int64_t)gridDim.x < n_items; ++k) {
            const int64_t idx = snake_item(k);
            if (idx >= n_items) continue;
            I = geom(idx);
            if (cap_report && I.cap_err) report(status, FOCUS_ERR_CAPACITY);
            if (I.valid) break;
        }
        return I;
    };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // ---- setup (once per CTA) -------------------------------------------------
    if (threadIdx.x == 0) {
        mbar_init(smem_addr(&bars->q), 1);
        mbar_init(smem_addr(&bars->q_free), 1);
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_addr(&bars->kv_full[s]), 1);
            mbar_init(smem_addr(&bars->kv_empty[s]), 1);
        }
        for (int t = 0; t < 2; ++t) {
            mbar_init(smem_addr(&bars->s_full[t]), 1);
            mbar_init(smem_addr(&bars->p_full[t]), BM);
            mbar_init(smem_addr(&bars->o_full[t]), 1);
            mbar_init(smem_addr(&bars->o_free[t]), BM);
        }
        mbar_init(smem_addr(&bars->drain), 1);
        bars->abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(&bars->tmem), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem;

    if constexpr (ROPE) {
        // prologue: all six 64-thread groups of every CTA rotate the first
        // rope_pro_heads K/V heads' units (their K and Q rows) at the full rate of the
        // SM, so that the attention can start on them while warps 2-3 go on with the
        // rest; shared scratch in the K/V stages, which no copy has touched yet
        const RopeSpan<D> rs{rope.t.theta, q_src, k_src, q_rot, k_rot, rot_done, T_span, q_per_kv,
                             win_off[w_begin], BHk};
        const int grp = threadIdx.x >> 6;
        rs.run((int32_t)blockIdx.x * (kThreads / 64) + grp, rs.n_chunks() * rope_pro_heads,
               (int32_t)gridDim.x * (kThreads / 64), threadIdx.x & 63, 1 + grp,
               reinterpret_cast<float2*>(smem + C::kSlotOff + grp * kRopeGroupScratch));
        __syncthreads();                               // the stage scratch is free for the copies
    }

    if (warp < 4) {
        setmaxnreg_dec<kRegsIssue<ROPE>>();
        if (warp == 0 && lane == 0) {
            // ============================================= TMA producer
            prefetch_tmap(&tm_q);
            prefetch_tmap(&tm_k);
            prefetch_tmap(&tm_v);
            prefetch_tmap(&tm_rk);
            prefetch_tmap(&tm_rv);
            const uint32_t bq = smem_addr(&bars->q);
            int64_t n_issued = 0;                        // K/V groups issued (one per MMA iteration), across items
            int it = 0;                                  // valid items started
            bool ok = true;
            int32_t ready_bh = -1;                       // ROPE: last head seen fully rotated
            int64_t k = 0;
            ItemGeom I = next_valid(k, true);
            while (ok && I.valid && !aborted(bars)) {
                int64_t kn = k + 1;
                ItemGeom N;
                N.valid = false;
                // the Q buffers are free once every QK MMA of the previous item has completed
                if (it > 0 && !mbar_wait(smem_addr(&bars->q_free), (it - 1) & 1, kWaitNs)) {
                    fail(bars, status);
                    break;
                }
                if constexpr (ROPE) {
                    // this head's rotated Q and K rows are all in the workspace
                    if (I.bh != ready_bh) {
                        if (!wait_count(rot_done + I.bh, (int32_t)((T_span + 63) / 64), kWaitNs)) {
                            fail(bars, status);
                            break;
                        }
                        ready_bh = I.bh;
                    }
                }
                mbar_expect_tx(bq, 2 * C::kTileBytes);
                const int32_t qrow = GQA ? I.bh * q_per_kv + I.member : I.bh;
                for (int t = 0; t < 2; ++t)
                    load_tile<D>(smem_addr(smem + C::kQOff + t * C::kTileBytes), &tm_q, I.row_base + I.a0 + t * BM,
                                 qrow, bq);
                // group g = {V_{g-1}, K_g}: everything MMA iteration g reads, in one stage
                for (int g = 0; g <= I.n_kv_max; ++g) {
                    const int64_t n = n_issued;
                    const int st = (int)(n & 1);
                    const int64_t use = n >> 1;
                    if (use > 0 && !mbar_wait(smem_addr(&bars->kv_empty[st]), (uint32_t)((use - 1) & 1), kWaitNs)) {
                        fail(bars, status);
                        ok = false;
                        break;
                    }
                    const uint32_t bf = smem_addr(&bars->kv_full[st]);
                    mbar_expect_tx(bf, (uint32_t)(((g >= 1) + (g < I.n_kv_max)) * C::kTileBytes));
                    const uint32_t sbase = smem_addr(smem + C::kSlotOff + 2 * st * C::kTileBytes);
                    if (g >= 1) {
                        const int jv = g - 1;
                        const bool ring = jv < I.n_ring;
                        const int32_t row = ring ? jv * BN : I.row_base + (jv - I.n_ring) * BN;
                        load_tile<D>(sbase, ring ? &tm_rv : &tm_v, row, I.bh, bf);
                    }
                    if (g < I.n_kv_max) {
                        const bool ring = g < I.n_ring;
                        const int32_t row = ring ? g * BN : I.row_base + (g - I.n_ring) * BN;
                        load_tile<D>(sbase + C::kTileBytes, ring ? &tm_rk : &tm_k, row, I.bh, bf);
                    }
                    n_issued = n + 1;
                    if (g == 0) {
                        // the next item, and its Q tiles into L2 while this item runs
                        N = next_valid(kn, true);
                        if (N.valid) {
                            const int32_t nq = GQA ? N.bh * q_per_kv + N.member : N.bh;
                            for (int t = 0; t < 2; ++t)
#pragma unroll
                                for (int x = 0; x < D / 64; ++x)
                                    tma_prefetch_3d(&tm_q, x * 64, N.row_base + N.a0 + t * BM, nq);
                        }
                    }
                }
                ++it;
                I = N;
                k = kn;
            }
            // drain: every issued copy must land before the CTA can exit
            if (it > 0) mbar_wait(bq, (it - 1) & 1, kWaitNs);
            for (int64_t n = (n_issued > 2 ? n_issued - 2 : 0); n < n_issued; ++n)
                mbar_wait(smem_addr(&bars->kv_full[n & 1]), (uint32_t)((n >> 1) & 1), kWaitNs);
        } else if (warp == 1 && lane == 0) {
            // ============================================= MMA issuer
            const uint32_t sq = smem_addr(smem + C::kQOff);
            const uint32_t sslot = smem_addr(smem + C::kSlotOff);
            int64_t nt0 = 0;                 // K/V groups consumed before this item
            int it = 0;                      // valid items
            int pc[2] = {0, 0};              // P tiles consumed per Q tile (p_full phases)
            int oc[2] = {0, 0};              // items with an epilogue per Q tile (o_free phases)
            bool ok = true;
            for (int64_t k = 0; ok && k * (int64_t)gridDim.x < n_items && !aborted(bars); ++k) {
                const int64_t idx = snake_item(k);
                if (idx >= n_items) continue;
                const ItemGeom I = geom(idx);
                if (!I.valid) continue;
                if (!mbar_wait(smem_addr(&bars->q), it & 1, kWaitNs)) { ok = false; break; }
                for (int j = 0; ok && j <= I.n_kv_max; ++j) {
                    const int64_t n = nt0 + j;                 // this iteration's group
                    const int st = (int)(n & 1);
                    if (!mbar_wait(smem_addr(&bars->kv_full[st]), (uint32_t)((n >> 1) & 1), kWaitNs)) {
                        ok = false;
                        break;
                    }
                    const uint32_t vbase = sslot + 2 * st * C::kTileBytes, kbase = vbase + C::kTileBytes;
                    tc_fence_after();
                    for (int t = 0; t < 2; ++t) {
                        const int nkt = t == 0 ? I.n_kv0 : I.n_kv1;
                        if (j >= 1 && j - 1 < nkt) {              // O_t += P_t(j-1) V_{j-1}
                            // the first PV of an item overwrites O_t: the previous item's
                            // epilogue must have read it
                            if (j == 1 && oc[t] > 0 &&
                                !mbar_wait(smem_addr(&bars->o_free[t]), (oc[t] - 1) & 1, kWaitNs)) {
                                ok = false;
                                break;
                            }
                            if (!mbar_wait(smem_addr(&bars->p_full[t]), pc[t] & 1, kWaitNs)) { ok = false; break; }
                            ++pc[t];
                            tc_fence_after();
                            issue_pv<D>(tmem + 256 + t * D, tmem + t * 128, vbase, j - 1 > 0);
                            if (j - 1 == nkt - 1) {
                                mma_commit(smem_addr(&bars->o_full[t]));
                                ++oc[t];
                            }
                        }
                        if (j < nkt) {                           // S_t = Q_t K_j^T
                            issue_qk<D>(tmem + t * 128, sq + t * C::kTileBytes, kbase);
                            mma_commit(smem_addr(&bars->s_full[t]));
                        }
                    }
                    if (!ok) break;
                    if (j == I.n_kv_max - 1) mma_commit(smem_addr(&bars->q_free));   // last QK of the item issued
                    mma_commit(smem_addr(&bars->kv_empty[st]));
                }
                nt0 += I.n_kv_max + 1;
                ++it;
            }
            if (!ok) fail(bars, status);
            // drain: all issued MMAs complete before TMEM is freed
            mma_commit(smem_addr(&bars->drain));
            mbar_wait(smem_addr(&bars->drain), 0, kWaitNs);
        } else if (ROPE && (warp == 2 || warp == 3)) {
            // ============================================= rotary embedding of the span
            if constexpr (ROPE) {
                const RopeSpan<D> rs{rope.t.theta, q_src, k_src, q_rot, k_rot, rot_done, T_span, q_per_kv,
                                     win_off[w_begin], BHk};
                const int32_t p0 = rs.n_chunks() * rope_pro_heads;   // the prologue's heads
                rs.run(p0 + (int32_t)blockIdx.x, rs.n_chunks() * BHk, (int32_t)gridDim.x, threadIdx.x - 64, 7,
                       reinterpret_cast<float2*>(smem + C::kRopeScratchOff));
            }
        }
    } else {
        // ================================================= softmax / epilogue
        setmaxnreg_inc<kRegsSoftmax<ROPE>>();
        const int t = (warp - 4) >> 2;                    // 0: warps 4-7, 1: warps 8-11
        const int quarter = warp & 3;                     // TMEM lanes this warp may access
        const int r = quarter * 32 + lane;                // row within the Q tile
        const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
        const uint32_t s_addr = tmem + lane_addr + t * 128;
        const uint32_t o_addr = tmem + lane_addr + 256 + t * D;
        int sc = 0, oc = 0;                               // s_full / o_full phases
        bool ok = true;
        for (int64_t k = 0; ok && k * (int64_t)gridDim.x < n_items && !aborted(bars); ++k) {
            const int64_t idx = snake_item(k);
            if (idx >= n_items) continue;
            const ItemGeom I = geom(idx);
            if (!I.valid) continue;
            const int n_kv = t == 0 ? I.n_kv0 : I.n_kv1;
            if (n_kv == 0) continue;
            const int qt = 2 * I.cta + t;                 // q-tile index within the window
            float m_run = -INFINITY, l_run = 0.f;
            for (int j = 0; j < n_kv; ++j) {
                if (!mbar_wait(smem_addr(&bars->s_full[t]), sc & 1, kWaitNs)) { ok = false; break; }
                ++sc;
                tc_fence_after();
                uint32_t sr[128];
                tmem_ld32(s_addr + 0, sr);
                tmem_ld32(s_addr + 32, sr + 32);
                tmem_ld32(s_addr + 64, sr + 64);
                tmem_ld32(s_addr + 96, sr + 96);
                tmem_wait_ld();
                float* s = reinterpret_cast<float*>(sr);
                // analytic mask: the ring's last partial tile and the diagonal window tile
                if (j < I.n_ring) {
                    const int lim = I.Rw - j * BN;        // keys [0, lim) of this tile are visible
                    if (lim < BN) {
#pragma unroll
                        for (int c = 0; c < BN; ++c)
                            if (c >= lim) s[c] = -INFINITY;
                    }
                } else if (j - I.n_ring == qt) {          // key c visible iff c <= r
#pragma unroll
                    for (int c = 0; c < BN; ++c)
                        if (c > r) s[c] = -INFINITY;
                }
                softmax_tile<D, false>(s, s_addr, o_addr, scale_log2, m_run, l_run, j > 0);
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(smem_addr(&bars->p_full[t]));
            }
            if (!ok) {
                fail(bars, status);
                break;
            }
            // ---- epilogue: O / l -> bf16 through a per-warp staging buffer (the Q
            // buffer may already hold the next item's Q), LSE; O_t is then free for
            // the next item's first PV. The item geometry is recomputed here from an
            // opaque copy of its index, so none of it stays live across the loop.
            int64_t idx_e = idx;
            asm volatile("mov.b64 %0, %0;" : "+l"(idx_e));
            const ItemGeom E = geom(idx_e);
            const int32_t aq = E.a0 + t * BM + r;         // in-window row
            ok = mbar_wait(smem_addr(&bars->o_full[t]), oc & 1, kWaitNs);
            ++oc;
            if (!ok) {
                fail(bars, status);
                break;
            }
            tc_fence_after();
            const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
            const int32_t bhq = GQA ? E.bh * q_per_kv + E.member : E.bh;   // Q, O and LSE rows
            // each warp stages a 32-column chunk of its 32 rows (64 B per row, 16-byte
            // pieces swizzled by row so both the row writes and the coalesced reads
            // are conflict-free), then stores 8 rows x 64 B per instruction
            uint8_t* stage = smem + C::kStageOff + (warp - 4) * 2048;
            __nv_bfloat16* otile = o + ((int64_t)bhq * T_span + E.row_base + E.a0 + t * BM + quarter * 32) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t orr[32];
                tmem_ld32(o_addr + c * 32, orr);
                tmem_wait_ld();
                if (c == D / 32 - 1) {                    // all of O_t read: release it
                    tc_fence_before();
                    mbar_arrive(smem_addr(&bars->o_free[t]));
                }
                const uint64_t il2 = f2_pack(inv_l, inv_l);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {              // O / l, scaled in pairs
                    uint32_t w4[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        float lo, hi;
                        f2_unpack(f2_mul(f2_pack(__uint_as_float(orr[q4 * 8 + 2 * e]),
                                                 __uint_as_float(orr[q4 * 8 + 2 * e + 1])), il2), lo, hi);
                        w4[e] = pack_bf16x2(lo, hi);
                    }
                    *reinterpret_cast<uint4*>(stage + lane * 64 + ((q4 ^ ((lane >> 1) & 3)) << 4)) =
                        make_uint4(w4[0], w4[1], w4[2], w4[3]);
                }
                __syncwarp();
#pragma unroll
                for (int i = 0; i < 32; i += 8) {
                    const int rr = i + (lane >> 2), q4 = lane & 3;
                    if (E.a0 + t * BM + quarter * 32 + rr < E.Tw)
                        *reinterpret_cast<uint4*>(otile + (int64_t)rr * D + c * 32 + q4 * 8) =
                            *reinterpret_cast<const uint4*>(stage + rr * 64 + ((q4 ^ ((rr >> 1) & 3)) << 4));
                }
                __syncwarp();
            }
            if (lse && aq < E.Tw)
                lse[(int64_t)bhq * T_span + E.row_base + aq] = (m_run + __log2f(l_run)) * 0.69314718055994531f;
        }
    }

    // ---- teardown ------------------------------------------------------------
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// Workspace layout (ROPE): int32 rot_done[B H] (padded to 256 bytes), then the
// rotated Q [B][H g][T_span][d] and K [B][H][T_span][d], bf16.

// K/V heads rotated in the kernel's prologue by all warps (the rest by warps 2-3
// beside the attention). One: at 128 kb, 32 query heads of one K/V head each,
// one head took 2.907 ms per launch, 2 / 5 of the heads 2.97 ms and all of them
// 3.035 ms.
int32_t rope_prologue_heads(int64_t BH) { return BH < 1 ? 0 : 1; }

template <int D, bool GQA, bool ROPE>
cudaError_t launch_d(const focus_cache& c, const focus_prefill_args& a, int32_t* status, cudaStream_t stream) {
    const int64_t BH = (int64_t)c.B * c.H;
    const int32_t g = c.q_per_kv > 1 ? c.q_per_kv : 1;
    const void* qmap = a.q;
    const void* kmap = a.k;
    int32_t* rot_done = nullptr;
    uint4 *q_rot = nullptr, *k_rot = nullptr;
    cudaError_t e;
    if constexpr (ROPE) {
        char* ws = static_cast<char*>(a.workspace);
        rot_done = reinterpret_cast<int32_t*>(ws);
        q_rot = reinterpret_cast<uint4*>(ws + rope_counter_bytes(c));
        k_rot = q_rot + BH * g * a.T_span * D / 8;
        qmap = q_rot;
        kmap = k_rot;
        if ((e = cudaMemsetAsync(rot_done, 0, (size_t)BH * 4, stream)) != cudaSuccess) return e;
    }
    CUtensorMap tq, tk, tv, trk, trv;
    if ((e = make_map(&tq, qmap, D, a.T_span, BH * g)) != cudaSuccess) return e;
    if ((e = make_map(&tk, kmap, D, a.T_span, BH)) != cudaSuccess) return e;
    if ((e = make_map(&tv, a.v, D, a.T_span, BH)) != cudaSuccess) return e;
    if (c.C_ring > 0) {
        if ((e = make_map(&trk, c.ring_k, D, c.C_ring, BH)) != cudaSuccess) return e;
        if ((e = make_map(&trv, c.ring_v, D, c.C_ring, BH)) != cudaSuccess) return e;
    } else {                                   // no ring: the maps are never read
        trk = tk;
        trv = tv;
    }
    const int smem = ROPE ? Cfg<D>::kSmemPersistentRope : Cfg<D>::kSmemPersistent;
    auto* kernel = prefill_tc_persistent_kernel<D, GQA, ROPE>;
    if ((e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
        return e;
    // the register split needs the launch registers it was sized for: with fewer,
    // the softmax warpgroups' setmaxnreg.inc could never be served
    cudaFuncAttributes fa;
    if ((e = cudaFuncGetAttributes(&fa, kernel)) != cudaSuccess) return e;
    if (fa.numRegs < kLaunchRegs) return cudaErrorInvalidConfiguration;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const int ctas_pw = (a.max_rows + 2 * BM - 1) / (2 * BM);
    // one CTA per SM, each walking every gridDim.x-th work item
    const int64_t n_items = (int64_t)(a.w_end - a.w_begin) * ctas_pw * g * c.H * c.B;
    RopeArg<ROPE> rope;
    if constexpr (ROPE) rope_table_fill(&rope.t, D, c.rope_theta);
    else rope.unused = 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(n_items < sms ? n_items : sms));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    // ROPE: a CTA's producer waits for rows that the other CTAs' rotating warps
    // write, so every CTA must be resident at once: a cooperative launch
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = ROPE ? 1 : 0;
    e = cudaLaunchKernelEx(&cfg, kernel, tq, tk, tv, trk, trv, (__nv_bfloat16*)a.o, a.lse, a.T_span, a.d_win_off,
                           a.d_ring_off, a.w_begin, a.w_end, ctas_pw, c.H, c.C_ring,
                           a.scale * 1.4426950408889634f, status, g, n_items, rope,
                           (const uint4*)a.q, (const uint4*)a.k, q_rot, k_rot, rot_done, (int32_t)BH,
                           rope_prologue_heads(BH));
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

size_t rope_counter_bytes(const focus_cache& c) { return ((size_t)c.B * c.H * 4 + 255) & ~(size_t)255; }

size_t persistent_workspace_bytes(const focus_cache& c, const focus_prefill_args& a) {
    if (!(c.rope_theta > 0.f)) return 0;
    const size_t g = c.q_per_kv > 1 ? (size_t)c.q_per_kv : 1;
    return rope_counter_bytes(c) + (size_t)c.B * c.H * (g + 1) * (size_t)a.T_span * c.d * 2;
}

cudaError_t launch_prefill_tc_persistent(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                                         cudaStream_t stream) {
    const bool gqa = c.q_per_kv > 1, rope = c.rope_theta > 0.f;
    if (c.d == 128) {
        if (rope) return gqa ? launch_d<128, true, true>(c, a, status, stream) : launch_d<128, false, true>(c, a, status, stream);
        return gqa ? launch_d<128, true, false>(c, a, status, stream) : launch_d<128, false, false>(c, a, status, stream);
    }
    if (rope) return gqa ? launch_d<64, true, true>(c, a, status, stream) : launch_d<64, false, true>(c, a, status, stream);
    return gqa ? launch_d<64, true, false>(c, a, status, stream) : launch_d<64, false, false>(c, a, status, stream);
}

}  // namespace prefill
}  // namespace focus
