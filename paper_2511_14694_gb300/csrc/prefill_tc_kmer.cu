// k-mer-local prefill (Sec. 3.2 "Visibility and summarization rule") with query
// tiles cut at k-mer boundaries, on the tcgen05 tensor cores.
//
// What it computes (the same rows as the k-mer-local mode of prefill_tc.cu): row
// a of window w, in k-mer c = a / (k_w + 1) (the whole window is one k-mer when
// k_w = 0 or k_w >= T_w), sees the earlier rows of its own k-mer and itself, the
// FOCUS rows of k-mers 0..c-1 of window w and the carried boundary (the last
// FOCUS row of window w-1), i.e. ring rows [ring_off[w] - b, ring_off[w] + c)
// (b = 1 when window w-1 kept rows: compaction runs before this call) and window
// rows [c (k_w + 1), a].
//
// Tiling: a work item is one query tile of kpt = (128 - RB) / (k_w + 1) whole
// k-mers of one (sequence, head, window) (RB: ring rows per tile, a multiple of 8
// chosen on the host so that every tile's ring rows fit). Every key such a tile
// sees fits one 128-row K/V tile: rows [0, RB) are ring rows from
// ring_off[w] - b (one TMA box of RB rows), rows [RB, 128) the window rows from
// the tile's first row (one box of 128 - RB rows), both boxes landing in one
// 128-byte-swizzled tile (RB * 128 bytes is a whole number of 1024-byte swizzle
// atoms). So each item is one QK MMA group, one softmax over one S tile and one PV
// group: no K/V tile of the 128-row grid that is mostly masked, no online-softmax
// iterations.
//
// Persistent: one CTA per SM walks the items; items alternate between two slots
// t (Q, K and V buffers, S_t and O_t in TMEM each), so that the loads and the
// epilogue of one item overlap the MMAs and softmax of the other:
//   warp 0     TMA producer: item i's Q and K once slot t's previous QK has
//              completed, its V once that item's PV has completed
//   warp 1     TMEM owner + MMA issuer: QK of item i, then PV of item i - 1
//   warps 2-3  idle; with the rotary embedding (ROPE) they rotate each item's Q
//              tile and the window rows of its K tile in shared memory, between
//              their TMA arrival and the item's QK (q and k rows are each read by
//              one item per query head here, so the rotation adds no HBM traffic;
//              the ring rows arrive rotated). A window row's position is
//              win_off[w] + its in-window row, and the K tile's window rows start
//              at the Q tile's first row, so Q row m and K row RB + m share every
//              angle.
//   warps 4-7 / 8-11  softmax + epilogue of the items of slot 0 / slot 1
// Every mbarrier wait is bounded; on timeout the kernel reports
// FOCUS_ERR_TIMEOUT, drains its own copies/MMAs (bounded), frees TMEM, returns.
#include "prefill_tc_common.cuh"

namespace focus {
namespace prefill {
namespace {

// register split: warpgroup 0 (TMA, MMA and, with the rotary embedding, the
// rotating warps 2-3) and the two softmax warpgroups
template <bool ROPE>
constexpr int kRegsIssue = ROPE ? 152 : 72;
template <bool ROPE>
constexpr int kRegsSoftmax = ROPE ? 176 : 216;
constexpr int64_t kKmerMaxRingRows = 64;   // ring rows a tile may hold (the window box keeps >= 64 rows)
constexpr int64_t kKmerMinItems = 2048;    // work items a launch needs for this kernel (~13 per SM)
static_assert(128 * kRegsIssue<false> + 256 * kRegsSoftmax<false> <= kThreads * kLaunchRegs, "register split over budget");
static_assert(128 * kRegsIssue<true> + 256 * kRegsSoftmax<true> <= kThreads * kLaunchRegs, "register split over budget");

struct KBars {
    uint64_t ld_qk[2];   // Q and K of the slot's item landed
    uint64_t ld_v[2];    // V landed
    uint64_t qk_free[2]; // the slot's QK completed: Q and K buffers reusable
    uint64_t v_free[2];  // the slot's PV completed: V buffer reusable
    uint64_t s_full[2];
    uint64_t p_full[2];
    uint64_t o_full[2];
    uint64_t o_free[2];  // the epilogue has read O_t
    uint64_t rot[2];     // ROPE: the slot's Q tile and K window rows are rotated
    uint64_t drain;
    uint32_t tmem;
    int32_t abort;
};
static_assert(sizeof(KBars) <= 256, "barriers must fit their 256-byte slot");

template <int D>
struct KCfg {
    static constexpr int kTile = Cfg<D>::kTileBytes;
    static constexpr int kQOff = 0;                  // Q_0, Q_1
    static constexpr int kKOff = 2 * kTile;          // K_0, K_1
    static constexpr int kVOff = 4 * kTile;          // V_0, V_1
    static constexpr int kBarOff = 6 * kTile;
    static constexpr int kStageOff = kBarOff + 256;  // O staging: 8 warps x 32 rows x 64 B
    static constexpr int kRopeOff = kStageOff + 8 * 2048;  // ROPE: the item's start angles, 64 x float2
    static constexpr int kSmem = kRopeOff + 512 + 1024;
};

// Position in the item space (sequence b, K/V head h, window w, query tile,
// query head of the group innermost) and the current window's data. A CTA walks
// a contiguous block of items, so the cursor moves by one (carrying into the
// next tile, window, head, sequence) and reads a window's offsets and cadence
// only when it enters it: the items are single MMA iterations, so per-item index
// arithmetic would cost as much as the work.
struct KCursor {
    int32_t b, h, w, tile, member;
    int32_t Tw, kdiv, nq, Rw, bnd, row_base;
    bool win_ok;

    __device__ __forceinline__ void enter_window(const int32_t* __restrict__ win_off,
                                                 const int32_t* __restrict__ ring_off,
                                                 const int32_t* __restrict__ k_per_window, int32_t w_begin,
                                                 int32_t w_end, int32_t RB, int32_t C_ring, int64_t T_span,
                                                 int32_t* status, bool report_errors) {
        const int32_t w0 = win_off[w_begin], wf = win_off[w];
        Tw = win_off[w + 1] - wf;
        row_base = wf - w0;
        const int32_t kw = k_per_window[w];
        kdiv = (kw > 0 && kw < Tw ? kw : Tw) + 1;
        const int32_t kpt = (128 - RB) / kdiv;
        nq = kpt * kdiv;
        Rw = ring_off[w];
        bnd = (w >= 1 && ring_off[w - 1] < Rw) ? 1 : 0;
        win_ok = kpt >= 1 && Tw > 0;
        if (!win_ok) {
            // the device schedule has a k-mer longer than the host's copy allowed for
            if (report_errors && Tw > 0) report(status, FOCUS_ERR_INVALID_ARG);
            return;
        }
        const int32_t c_max = (Tw - 1) / kdiv;      // the k-mer of the window's last row
        if (c_max + bnd > RB) {                     // more ring rows than a tile holds
            if (report_errors) report(status, FOCUS_ERR_INVALID_ARG);
            win_ok = false;
        } else if (Rw + c_max > C_ring || (int64_t)(win_off[w_end] - w0) > T_span) {
            if (report_errors) report(status, FOCUS_ERR_CAPACITY);
            win_ok = false;
        }
    }
    __device__ __forceinline__ int32_t s() const { return tile * nq; }
    __device__ __forceinline__ bool valid() const { return win_ok && tile * nq < Tw; }
    __device__ __forceinline__ int32_t rows() const { return nq < Tw - tile * nq ? nq : Tw - tile * nq; }
};

// Barrier `id` over `count` threads that also ORs a predicate over them: every
// participating thread gets the same result.
__device__ __forceinline__ bool named_bar_or(uint32_t id, uint32_t count, bool pred) {
    uint32_t r;
    asm volatile(
        "{\n .reg .pred p, q;\n setp.ne.u32 q, %1, 0;\n bar.red.or.pred p, %2, %3, q;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(r)
        : "r"((uint32_t)pred), "r"(id), "r"(count)
        : "memory");
    return r != 0;
}

template <int D, bool GQA, bool ROPE>
__global__ void __launch_bounds__(kThreads, 1) prefill_tc_kmer_kernel(
        const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kw,
        const __grid_constant__ CUtensorMap tm_vw, const __grid_constant__ CUtensorMap tm_rk,
        const __grid_constant__ CUtensorMap tm_rv, __nv_bfloat16* __restrict__ o, float* __restrict__ lse,
        int64_t T_span, const int32_t* __restrict__ win_off, const int32_t* __restrict__ ring_off,
        const int32_t* __restrict__ k_per_window, int32_t w_begin, int32_t w_end, int32_t max_tiles, int32_t RB,
        int32_t H, int32_t C_ring, float scale_log2, int32_t* status, int32_t q_per_kv, int64_t n_items,
        const __grid_constant__ RopeArg<ROPE> rope) {
    using C = KCfg<D>;
    extern __shared__ unsigned char smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    KBars* bars = reinterpret_cast<KBars*>(smem + C::kBarOff);
    if (*(volatile int32_t*)status == FOCUS_ERR_TIMEOUT) return;
    // this CTA's block of the item space [i0, i1)
    const int64_t i0 = n_items * blockIdx.x / gridDim.x, i1 = n_items * (blockIdx.x + 1) / gridDim.x;
    const int32_t g = GQA ? q_per_kv : 1;
    auto start = [&](bool report_errors) {
        KCursor c;
        const int64_t per_w = (int64_t)max_tiles * g, per_head = per_w * (w_end - w_begin);
        int64_t x = i0;
        c.member = (int32_t)(x % g);
        c.tile = (int32_t)((x / g) % max_tiles);
        c.w = w_begin + (int32_t)((x / per_w) % (w_end - w_begin));
        c.h = (int32_t)((x / per_head) % H);
        c.b = (int32_t)(x / (per_head * H));
        if (i0 < i1)
            c.enter_window(win_off, ring_off, k_per_window, w_begin, w_end, RB, C_ring, T_span, status, report_errors);
        return c;
    };
    auto advance = [&](KCursor& c, bool report_errors) {
        if (++c.member < g) return;
        c.member = 0;
        if (++c.tile < max_tiles) return;
        c.tile = 0;
        if (++c.w == w_end) {
            c.w = w_begin;
            if (++c.h == H) {
                c.h = 0;
                ++c.b;
            }
        }
        c.enter_window(win_off, ring_off, k_per_window, w_begin, w_end, RB, C_ring, T_span, status, report_errors);
    };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t ring_box_bytes = (uint32_t)RB * 128, win_box_bytes = (uint32_t)(128 - RB) * 128;

    if (threadIdx.x == 0) {
        for (int t = 0; t < 2; ++t) {
            mbar_init(smem_addr(&bars->ld_qk[t]), 1);
            mbar_init(smem_addr(&bars->ld_v[t]), 1);
            mbar_init(smem_addr(&bars->qk_free[t]), 1);
            mbar_init(smem_addr(&bars->v_free[t]), 1);
            mbar_init(smem_addr(&bars->s_full[t]), 1);
            mbar_init(smem_addr(&bars->p_full[t]), BM);
            mbar_init(smem_addr(&bars->o_full[t]), 1);
            mbar_init(smem_addr(&bars->o_free[t]), BM);
            mbar_init(smem_addr(&bars->rot[t]), 1);
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
    auto fail_k = [&]() {
        report(status, FOCUS_ERR_TIMEOUT);
        atomicExch(&bars->abort, 1);
    };
    auto aborted_k = [&]() { return *(volatile int32_t*)&bars->abort != 0; };

    if (warp < 4) {
        setmaxnreg_dec<kRegsIssue<ROPE>>();
        if (warp == 0 && lane == 0) {
            // ============================================= TMA producer
            prefetch_tmap(&tm_q);
            prefetch_tmap(&tm_kw);
            prefetch_tmap(&tm_vw);
            prefetch_tmap(&tm_rk);
            prefetch_tmap(&tm_rv);
            int64_t i = 0;                                   // valid items (slot t = i & 1)
            KCursor I = start(true);
            for (int64_t idx = i0; idx < i1 && !aborted_k(); ++idx, advance(I, true)) {
                if (!I.valid()) continue;
                const int t = (int)(i & 1);
                const int64_t u = i >> 1;                    // items of slot t before this one
                if (u > 0 && !mbar_wait(smem_addr(&bars->qk_free[t]), (uint32_t)((u - 1) & 1), kWaitNs)) {
                    fail_k();
                    break;
                }
                const uint32_t bqk = smem_addr(&bars->ld_qk[t]);
                mbar_expect_tx(bqk, (uint32_t)(C::kTile + (D / 64) * (ring_box_bytes + win_box_bytes)));
                const int32_t bh = I.b * H + I.h;
                const int32_t qrow = GQA ? bh * q_per_kv + I.member : bh;
                const int32_t row = I.row_base + I.s();
                load_tile<D>(smem_addr(smem + C::kQOff + t * C::kTile), &tm_q, row, qrow, bqk);
                const uint32_t kt = smem_addr(smem + C::kKOff + t * C::kTile);
#pragma unroll
                for (int xh = 0; xh < D / 64; ++xh) {
                    tma_load_3d(kt + xh * kBoxBytes, &tm_rk, xh * 64, I.Rw - I.bnd, bh, bqk);
                    tma_load_3d(kt + xh * kBoxBytes + ring_box_bytes, &tm_kw, xh * 64, row, bh, bqk);
                }
                if (u > 0 && !mbar_wait(smem_addr(&bars->v_free[t]), (uint32_t)((u - 1) & 1), kWaitNs)) {
                    fail_k();
                    break;
                }
                const uint32_t bv = smem_addr(&bars->ld_v[t]);
                mbar_expect_tx(bv, (uint32_t)((D / 64) * (ring_box_bytes + win_box_bytes)));
                const uint32_t vt = smem_addr(smem + C::kVOff + t * C::kTile);
#pragma unroll
                for (int xh = 0; xh < D / 64; ++xh) {
                    tma_load_3d(vt + xh * kBoxBytes, &tm_rv, xh * 64, I.Rw - I.bnd, bh, bv);
                    tma_load_3d(vt + xh * kBoxBytes + ring_box_bytes, &tm_vw, xh * 64, row, bh, bv);
                }
                ++i;
            }
            // drain: the last item of each slot has landed before the CTA can exit
            for (int64_t j = (i > 2 ? i - 2 : 0); j < i; ++j) {
                mbar_wait(smem_addr(&bars->ld_qk[j & 1]), (uint32_t)((j >> 1) & 1), kWaitNs);
                mbar_wait(smem_addr(&bars->ld_v[j & 1]), (uint32_t)((j >> 1) & 1), kWaitNs);
            }
        } else if (warp == 1 && lane == 0) {
            // ============================================= MMA issuer
            bool ok = true;
            int64_t i = 0;
            // PV of item j (slot t = j & 1): O_t = P_t V_t, once the item's V and P
            // are in and the epilogue of the slot's previous item has read O_t
            auto pv = [&](int64_t j) {
                const int t = (int)(j & 1);
                const int64_t u = j >> 1;
                if (!mbar_wait(smem_addr(&bars->ld_v[t]), (uint32_t)(u & 1), kWaitNs)) return false;
                if (!mbar_wait(smem_addr(&bars->p_full[t]), (uint32_t)(u & 1), kWaitNs)) return false;
                if (u > 0 && !mbar_wait(smem_addr(&bars->o_free[t]), (uint32_t)((u - 1) & 1), kWaitNs)) return false;
                tc_fence_after();
                issue_pv<D>(tmem + 256 + t * D, tmem + t * 128, smem_addr(smem + C::kVOff + t * C::kTile), false);
                mma_commit(smem_addr(&bars->o_full[t]));
                mma_commit(smem_addr(&bars->v_free[t]));
                return true;
            };
            KCursor I = start(false);
            for (int64_t idx = i0; ok && idx < i1 && !aborted_k(); ++idx, advance(I, false)) {
                if (!I.valid()) continue;
                const int t = (int)(i & 1);
                const int64_t u = i >> 1;
                // Q and K landed (and, with the rotary embedding, are rotated)
                if (!mbar_wait(smem_addr(ROPE ? &bars->rot[t] : &bars->ld_qk[t]), (uint32_t)(u & 1), kWaitNs)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                issue_qk<D>(tmem + t * 128, smem_addr(smem + C::kQOff + t * C::kTile),
                            smem_addr(smem + C::kKOff + t * C::kTile));
                mma_commit(smem_addr(&bars->s_full[t]));
                mma_commit(smem_addr(&bars->qk_free[t]));
                if (i >= 1 && !pv(i - 1)) {
                    ok = false;
                    break;
                }
                ++i;
            }
            if (ok && i >= 1 && !aborted_k()) ok = pv(i - 1);
            if (!ok) fail_k();
            mma_commit(smem_addr(&bars->drain));
            mbar_wait(smem_addr(&bars->drain), 0, kWaitNs);
        } else if (ROPE && (warp == 2 || warp == 3)) {
            // ============================================= rotary embedding (warps 2-3)
            if constexpr (ROPE) {
                // thread tau owns pair chunk jj (columns 8 jj .. and D/2 + 8 jj ..) of
                // rows g, g + G, ... of the item's Q tile and of its K tile's window rows
                constexpr int HALF = D / 16, G = 64 / HALF;
                const int tau = threadIdx.x - 64, jj = tau % HALF, gg = tau / HALF;
                float2* kb = reinterpret_cast<float2*>(smem + C::kRopeOff);
                float2 off[8];
                Rot8 step;
                rope_offsets(rope.t.theta, 8 * jj, gg, G, off, step);
                const double theta_own = tau < D / 2 ? rope.t.theta[tau] : 0.0;
                const int64_t w0 = win_off[w_begin];
                const int clo = 8 * jj, chi = 8 * jj + D / 2;
                int64_t i = 0;
                KCursor I = start(false);
                for (int64_t idx = i0; idx < i1; ++idx, advance(I, false)) {
                    if (!I.valid()) continue;
                    const int t = (int)(i & 1);
                    const int64_t u = i >> 1;
                    ++i;
                    const bool landed = mbar_wait(smem_addr(&bars->ld_qk[t]), (uint32_t)(u & 1), kWaitNs);
                    // position of the tile's first row; the item's start angles
                    if (landed && tau < D / 2) kb[tau] = rope_cs((double)(w0 + I.row_base + I.s()) * theta_own);
                    // one decision for all 64 threads: a bounded wait may give up in some only
                    if (named_bar_or(1, 64, !landed || aborted_k())) {
                        if (!landed) fail_k();
                        break;
                    }
                    float2 cs[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) cs[e] = rope_mul(kb[8 * jj + e], off[e]);
                    Rot8 rot = rot8_make(cs);
                    uint8_t* qt = smem + C::kQOff + t * C::kTile;
                    uint8_t* kt = smem + C::kKOff + t * C::kTile;
                    // the item's query rows and the window keys they can see (its own
                    // k-mers: window rows below s + rows)
                    const int n_rows = I.rows();
#pragma unroll 1
                    for (int m = gg; m < n_rows; m += G) {
                        const int rk = RB + m;
                        uint4* qlo = reinterpret_cast<uint4*>(qt + (clo / 64) * kBoxBytes + m * 128 +
                                                              ((((clo % 64) / 8) ^ (m & 7)) << 4));
                        uint4* qhi = reinterpret_cast<uint4*>(qt + (chi / 64) * kBoxBytes + m * 128 +
                                                              ((((chi % 64) / 8) ^ (m & 7)) << 4));
                        uint4* klo = reinterpret_cast<uint4*>(kt + (clo / 64) * kBoxBytes + rk * 128 +
                                                              ((((clo % 64) / 8) ^ (rk & 7)) << 4));
                        uint4* khi = reinterpret_cast<uint4*>(kt + (chi / 64) * kBoxBytes + rk * 128 +
                                                              ((((chi % 64) / 8) ^ (rk & 7)) << 4));
                        uint4 a = *qlo, b = *qhi, c = *klo, d = *khi;
                        rot8_apply(a, b, rot);
                        rot8_apply(c, d, rot);
                        *qlo = a;
                        *qhi = b;
                        *klo = c;
                        *khi = d;
                        rot8_step(rot, step);
                    }
                    fence_proxy_async_smem();             // the MMA reads these rows through the async proxy
                    named_bar_sync(1, 64);                 // every row rotated; kb free for the next item
                    if (tau == 0) mbar_arrive(smem_addr(&bars->rot[t]));
                }
            }
        }
    } else {
        // ================================================= softmax / epilogue
        setmaxnreg_inc<kRegsSoftmax<ROPE>>();
        const int t = (warp - 4) >> 2;                    // slot of this warpgroup
        const int quarter = warp & 3;
        const int r = quarter * 32 + lane;                // row within the Q tile
        const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
        const uint32_t s_addr = tmem + lane_addr + t * 128;
        const uint32_t o_addr = tmem + lane_addr + 256 + t * D;
        uint8_t* stage = smem + C::kStageOff + (warp - 4) * 2048;
        int64_t i = 0;
        bool ok = true;
        KCursor I = start(false);
        for (int64_t idx = i0; ok && idx < i1 && !aborted_k(); ++idx, advance(I, false)) {
            if (!I.valid()) continue;
            const int64_t mine = i;
            ++i;
            if ((mine & 1) != t) continue;                 // the other slot's item
            const int64_t u = mine >> 1;
            if (!mbar_wait(smem_addr(&bars->s_full[t]), (uint32_t)(u & 1), kWaitNs)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t sr[128];
            tmem_ld32(s_addr + 0, sr);
            tmem_ld32(s_addr + 32, sr + 32);
            tmem_ld32(s_addr + 64, sr + 64);
            tmem_ld32(s_addr + 96, sr + 96);
            tmem_wait_ld();
            float* sv = reinterpret_cast<float*>(sr);
            // row a of the window (k-mer c) sees key columns [0, c + bnd) (ring rows
            // ring_off[w] - bnd ..) and RB + [c kdiv - s, r] (its k-mer's rows up to itself)
            const int32_t a = I.s() + r;
            const int32_t c = a / I.kdiv;
            const int32_t ring_hi = c + I.bnd;
            const int32_t lo = RB + c * I.kdiv - I.s(), hi = RB + r;
#pragma unroll
            for (int col = 0; col < BN; ++col)
                if (col >= ring_hi && (col < lo || col > hi)) sv[col] = -INFINITY;
            float m_run = -INFINITY, l_run = 0.f;
            softmax_tile<D, true>(sv, s_addr, o_addr, scale_log2, m_run, l_run, false);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(smem_addr(&bars->p_full[t]));
            // ---- epilogue: O / l -> bf16 through the per-warp staging buffer, LSE
            ok = mbar_wait(smem_addr(&bars->o_full[t]), (uint32_t)(u & 1), kWaitNs);
            if (!ok) break;
            tc_fence_after();
            const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
            const int32_t bhq = (I.b * H + I.h) * g + I.member;       // Q, O and LSE rows
            const int32_t rows = I.rows();                             // rows of this tile to store
            const int64_t orow = (int64_t)bhq * T_span + I.row_base + I.s();
            __nv_bfloat16* otile = o + (orow + quarter * 32) * D;
#pragma unroll
            for (int cc = 0; cc < D / 32; ++cc) {
                uint32_t orr[32];
                tmem_ld32(o_addr + cc * 32, orr);
                tmem_wait_ld();
                if (cc == D / 32 - 1) {                    // all of O_t read: release it
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
                for (int k8 = 0; k8 < 32; k8 += 8) {
                    const int rr = k8 + (lane >> 2), q4 = lane & 3;
                    if (quarter * 32 + rr < rows)
                        *reinterpret_cast<uint4*>(otile + (int64_t)rr * D + cc * 32 + q4 * 8) =
                            *reinterpret_cast<const uint4*>(stage + rr * 64 + ((q4 ^ ((rr >> 1) & 3)) << 4));
                }
                __syncwarp();
            }
            if (lse && r < rows) lse[orow + r] = (m_run + __log2f(l_run)) * 0.69314718055994531f;
        }
        if (!ok) fail_k();
    }

    // ---- teardown ------------------------------------------------------------
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

template <int D, bool GQA, bool ROPE>
cudaError_t launch_d(const focus_cache& c, const focus_prefill_args& a, int32_t RB, int32_t max_tiles,
                     int32_t* status, cudaStream_t stream) {
    const int64_t BH = (int64_t)c.B * c.H;
    const int32_t g = c.q_per_kv > 1 ? c.q_per_kv : 1;
    CUtensorMap tq, tkw, tvw, trk, trv;
    cudaError_t e;
    if ((e = make_map(&tq, a.q, D, a.T_span, BH * g)) != cudaSuccess) return e;
    if ((e = make_map(&tkw, a.k, D, a.T_span, BH, 128 - RB)) != cudaSuccess) return e;
    if ((e = make_map(&tvw, a.v, D, a.T_span, BH, 128 - RB)) != cudaSuccess) return e;
    if (c.C_ring > 0) {
        if ((e = make_map(&trk, c.ring_k, D, c.C_ring, BH, RB)) != cudaSuccess) return e;
        if ((e = make_map(&trv, c.ring_v, D, c.C_ring, BH, RB)) != cudaSuccess) return e;
    } else {   // no ring: the ring rows are all masked, read any RB rows of k and v
        if ((e = make_map(&trk, a.k, D, a.T_span, BH, RB)) != cudaSuccess) return e;
        if ((e = make_map(&trv, a.v, D, a.T_span, BH, RB)) != cudaSuccess) return e;
    }
    const int smem = KCfg<D>::kSmem;
    auto* kernel = prefill_tc_kmer_kernel<D, GQA, ROPE>;
    if ((e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
        return e;
    cudaFuncAttributes fa;
    if ((e = cudaFuncGetAttributes(&fa, kernel)) != cudaSuccess) return e;
    if (fa.numRegs < kLaunchRegs) return cudaErrorInvalidConfiguration;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const int64_t n_items = (int64_t)(a.w_end - a.w_begin) * max_tiles * g * c.H * c.B;
    const dim3 grid((unsigned)(n_items < sms ? n_items : sms));
    RopeArg<ROPE> rope;
    if constexpr (ROPE) rope_table_fill(&rope.t, D, c.rope_theta);
    else rope.unused = 0;
    kernel<<<grid, kThreads, smem, stream>>>(tq, tkw, tvw, trk, trv, (__nv_bfloat16*)a.o, a.lse, a.T_span,
                                             a.d_win_off, a.d_ring_off, c.k_per_window, a.w_begin, a.w_end,
                                             max_tiles, RB, c.H, c.C_ring, a.scale * 1.4426950408889634f, status, g,
                                             n_items, rope);
    return cudaGetLastError();
}

}  // namespace

bool kmer_tiling(const focus_cache& c, const focus_prefill_args& a, int32_t* RB, int32_t* max_tiles) {
    if (!a.h_k_per_window || a.max_rows <= 0) return false;
    // ring rows a tile needs: the carried boundary + the FOCUS rows of its earlier
    // k-mers, at most one per k bases of the window (+1 for an open last k-mer)
    int64_t ring = 1, kdiv_max = 1;
    for (int32_t w = a.w_begin; w < a.w_end; ++w) {
        const int64_t k = a.h_k_per_window[w];
        if (k < 0) return false;
        const int64_t kdiv = (k > 0 && k < a.max_rows ? k : a.max_rows) + 1;
        const int64_t r = k > 0 ? (a.max_rows + k - 1) / k + 1 : 1;
        if (r > ring) ring = r;
        if (kdiv > kdiv_max) kdiv_max = kdiv;
    }
    const int64_t rb = (ring + 7) / 8 * 8;
    if (rb > kKmerMaxRingRows || kdiv_max > 128 - rb) return false;
    // tiles per window: a tile holds (128 - RB) / kdiv whole k-mers, which is not
    // monotonic in the k-mer length, so take the most over the windows (a device
    // k-mer is never longer than the host's bound here, so its tiles are no more)
    int64_t tiles = 1;
    for (int32_t w = a.w_begin; w < a.w_end; ++w) {
        const int64_t k = a.h_k_per_window[w];
        const int64_t kdiv = (k > 0 && k < a.max_rows ? k : a.max_rows) + 1;
        const int64_t nq = ((128 - rb) / kdiv) * kdiv;
        const int64_t t = (a.max_rows + nq - 1) / nq;
        if (t > tiles) tiles = t;
    }
    // a launch with few items (one window of a stream) does not fill the per-SM
    // pipelines of this persistent kernel: one 1 kb window at batch 4 (1,280
    // items) ran 50.8 us per launch against 47.3 for the one-CTA-per-item kernel
    const int64_t g = c.q_per_kv > 1 ? c.q_per_kv : 1;
    if ((int64_t)(a.w_end - a.w_begin) * tiles * g * c.H * c.B < kKmerMinItems) return false;
    *RB = (int32_t)rb;
    *max_tiles = (int32_t)tiles;
    return true;
}

cudaError_t launch_prefill_tc_kmer(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                                   cudaStream_t stream) {
    int32_t RB = 0, max_tiles = 0;
    if (!kmer_tiling(c, a, &RB, &max_tiles)) return cudaErrorInvalidValue;
    const bool gqa = c.q_per_kv > 1, rope = c.rope_theta > 0.f;
    if (c.d == 128) {
        if (rope)
            return gqa ? launch_d<128, true, true>(c, a, RB, max_tiles, status, stream)
                       : launch_d<128, false, true>(c, a, RB, max_tiles, status, stream);
        return gqa ? launch_d<128, true, false>(c, a, RB, max_tiles, status, stream)
                   : launch_d<128, false, false>(c, a, RB, max_tiles, status, stream);
    }
    if (rope)
        return gqa ? launch_d<64, true, true>(c, a, RB, max_tiles, status, stream)
                   : launch_d<64, false, true>(c, a, RB, max_tiles, status, stream);
    return gqa ? launch_d<64, true, false>(c, a, RB, max_tiles, status, stream)
               : launch_d<64, false, false>(c, a, RB, max_tiles, status, stream);
}

}  // namespace prefill
}  // namespace focus
