// Windowed prefill attention over the compressed context on the 5th-generation
// tensor cores (tcgen05.mma, accumulators in TMEM, operands staged by TMA).
//
// What it computes (Eq. focus-attn's visible set; App. A.1-A.2): row a of
// window w attends to ring rows [0, ring_off[w]) (retained FOCUS K/V of all
// earlier windows, fully visible) and to window rows [0, a] (causal). The mask
// is analytic per 128-key tile: only the last partial ring tile (key >= R_w)
// and the diagonal window tile (key > row) are masked.
//
// k-mer-local mode (LOCAL; Sec. 3.2 "Visibility and summarization rule"): row a
// of k-mer c = a / (k_w + 1) sees the rows [c (k_w + 1), a] of its own k-mer, the
// FOCUS rows of k-mers 0..c-1 of its window and the carried boundary (the last
// FOCUS row of window w-1). The ring already holds window w's own FOCUS rows
// right after the boundary, so the CTA reads ring rows
// [ring_off[w] - boundary, ring_off[w] + c_last) and window rows from the first
// row of its first k-mer to its last row; each row's visible keys are one
// interval per tile.
//
// CTA = two 128-row Q tiles of one (sequence, head, window) that share every
// K/V tile, 12 warps in three warpgroups:
//   warp 0     TMA producer: Q tiles once, then per MMA iteration j the group
//              {V_{j-1}, K_j} into one of two stages (one full/empty mbarrier pair
//              per stage, so the issuer waits once per iteration)
//   warp 1     TMEM owner + MMA issuer (one thread):
//                S_t = Q_t K_j^T            (SS, both operands K-major, SW128)
//                O_t += P_t V_j             (TS, P_t in TMEM over S_t, V MN-major)
//              in ping-pong order PV_0(j-1), QK_0(j), PV_1(j-1), QK_1(j)
//   warps 2-3  idle (they keep the softmax warpgroups aligned to warpgroups)
//   warps 4-7  softmax of tile 0, warps 8-11 softmax of tile 1: each thread owns
//              one row (32x32b TMEM loads), online softmax in the log2 domain with
//              lazy rescaling of O (only when the running max grows by > 8),
//              writes P (bf16) back into TMEM, and at the end normalises O and
//              stores O and the LSE.
// TMEM: S_0 cols [0,128), S_1 [128,256), O_0 [256, 256+D), O_1 [256+D, 256+2D).
//
// Rotary embedding (ROPE): the softmax warps rotate the two Q tiles in shared
// memory before the first S = Q K^T (q_rot barrier), and warps 2-3 rotate each
// window K tile between its stage's arrival and its MMA (k_rot, one per stage); ring tiles
// arrive rotated. Each rotating thread owns eight column pairs (i, i + d/2) of a
// set of rows spaced G apart: one fp64 angle per pair and tile (or 64-row
// segment) start, then the fixed per-row offsets of a host table.
// Every mbarrier wait is bounded; on timeout the kernel reports
// FOCUS_ERR_TIMEOUT, drains its own copies/MMAs (bounded), frees TMEM, returns.
#include <mutex>

#include "prefill_tc_common.cuh"

namespace focus {
namespace prefill {

// ---------------------------------------------------------------- tensor maps

namespace {

// One S row of a tile: 32 lanes x 128 consecutive 32-bit columns in one
// instruction (the four 32-column loads in one; the rotary variants keep those,
// which spill less next to their rotation code).
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, uint32_t* r) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x128.b32 {"
        "%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,"
        "%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
        "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,"
        "%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,"
        "%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,"
        "%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,"
        "%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127}, [%128];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
          "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
          "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
          "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
          "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]),
          "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]),
          "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]),
          "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]),
          "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]),
          "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]),
          "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]),
          "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]),
          "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
        : "r"(taddr));
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::mutex g_encode_mu;

cudaError_t get_encode(PFN_cuTensorMapEncodeTiled_v12000* out) {
    std::lock_guard<std::mutex> lock(g_encode_mu);
    if (!g_encode) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess) return e;
        if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    *out = g_encode;
    return cudaSuccess;
}

}  // namespace

// 3-D map over a [BH][rows][d] bf16 tensor, box = box_rows rows x 64 columns
// (a multiple of 8, <= 128), 128-byte swizzle.
cudaError_t make_map(CUtensorMap* m, const void* ptr, int d, int64_t rows, int64_t bh, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 enc;
    cudaError_t e = get_encode(&enc);
    if (e != cudaSuccess) return e;
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)rows, (cuuint64_t)bh};
    cuuint64_t strides[2] = {(cuuint64_t)d * 2, (cuuint64_t)d * 2 * (cuuint64_t)rows};
    cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, es,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace prefill

namespace {

using namespace prefill;

// Register split (variants without the rotary embedding): warpgroup 0 (TMA, MMA
// and two idle warps) gives registers back, the two softmax warpgroups take
// them: 128 x 72 + 256 x 216 = 128 x 56 + 256 x 224 = 384 x 168 (d = 128 issues
// twice the MMAs per tile and keeps its base descriptors live). With the rotary
// embedding warps 2-3 rotate K tiles and need their registers (every split tried
// spilled more than none), so those variants keep 168 each.
template <int D>
constexpr int kRegsIssue = D == 128 ? 72 : 56;
template <int D>
constexpr int kRegsSoftmax = D == 128 ? 216 : 224;
static_assert(128 * kRegsIssue<128> + 256 * kRegsSoftmax<128> <= kThreads * kLaunchRegs, "register split over budget");
static_assert(128 * kRegsIssue<64> + 256 * kRegsSoftmax<64> <= kThreads * kLaunchRegs, "register split over budget");

// Q/O/LSE row of this CTA's query head, read afresh from the block index where
// it is used (keeping it in a register across the softmax loop costs spills).
__device__ __forceinline__ int32_t query_head_row(int32_t H, int32_t q_per_kv) {
    uint32_t x, y, z;
    asm volatile("mov.u32 %0, %%ctaid.x;" : "=r"(x));
    asm volatile("mov.u32 %0, %%ctaid.y;" : "=r"(y));
    asm volatile("mov.u32 %0, %%ctaid.z;" : "=r"(z));
    return ((int32_t)z * H + (int32_t)y) * q_per_kv + (int32_t)(x % (uint32_t)q_per_kv);
}

template <int D, bool LOCAL, bool ROPE, bool GQA>
__global__ void __launch_bounds__(kThreads, 1) prefill_tc_kernel(
        const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
        const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_rk,
        const __grid_constant__ CUtensorMap tm_rv, __nv_bfloat16* __restrict__ o, float* __restrict__ lse,
        int64_t T_span, const int32_t* __restrict__ win_off, const int32_t* __restrict__ ring_off, int32_t w_begin,
        int32_t w_end, int32_t ctas_pw, int32_t H, int32_t C_ring, float scale_log2, int32_t* status,
        const int32_t* __restrict__ k_per_window, const __grid_constant__ RopeArg<ROPE> rope, int32_t q_per_kv) {
    using C = Cfg<D>;
    extern __shared__ unsigned char smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    Bars* bars = reinterpret_cast<Bars*>(smem + C::kBarOff);

    // ---- work item (longest first: later windows have longer rings) --------
    // GQA: the q_per_kv query heads that share a K/V head are adjacent in launch
    // order (a separate instantiation: the division costs registers elsewhere)
    const uint32_t item = GQA ? blockIdx.x / (uint32_t)q_per_kv : blockIdx.x;
    const int32_t member = GQA ? (int32_t)(blockIdx.x % (uint32_t)q_per_kv) : 0;
    const int32_t wi = item / ctas_pw;
    const int32_t cta = ctas_pw - 1 - (int32_t)(item % ctas_pw);
    const int32_t w = w_end - 1 - wi;
    const int h = blockIdx.y, b = blockIdx.z;     // h: K/V head
    const int32_t bh = b * H + h;                   // K/V and ring rows
    const int32_t w0 = win_off[w_begin];
    const int32_t Tw = win_off[w + 1] - win_off[w];
    const int32_t a0 = cta * 2 * BM;
    if (a0 >= Tw) return;                               // uniform: nothing allocated yet
    // Once any CTA has given up on a wait, later CTAs skip their work so that a
    // systematic stall costs one wave of bounded waits, not one per wave.
    if (*(volatile int32_t*)status == FOCUS_ERR_TIMEOUT) return;
    const int32_t Rw = ring_off[w];
    // LOCAL: k-mer length + 1 (a window without summaries, or with k >= T_w, is one
    // k-mer), boundary present?, key ranges [ring_lo, ...) and [win_lo, ...)
    int32_t kdiv = 1, bnd = 0, ring_lo = 0, win_lo = 0, ring_hi = Rw;
    int n_ring, n_win = 0, n_win0 = 0;
    if (LOCAL) {
        const int32_t kw = k_per_window[w];
        kdiv = (kw > 0 && kw < Tw ? kw : Tw) + 1;
        bnd = (w >= 1 && ring_off[w - 1] < Rw) ? 1 : 0;
        const int32_t a_last = (a0 + 2 * BM < Tw ? a0 + 2 * BM : Tw) - 1;
        ring_lo = Rw - bnd;
        ring_hi = Rw + a_last / kdiv;
        win_lo = (a0 / kdiv) * kdiv;
        n_ring = (ring_hi - ring_lo + BN - 1) / BN;
        n_win = (a_last + 1 - win_lo + BN - 1) / BN;
        // Q tile 0 ends at row a0 + BM - 1: its window keys are a prefix of the CTA's
        n_win0 = ((a0 + BM < Tw ? a0 + BM : Tw) - win_lo + BN - 1) / BN;
    } else {
        n_ring = (Rw + BN - 1) / BN;
    }
    if (ring_hi > C_ring || (int64_t)(win_off[w_end] - w0) > T_span) {
        if (threadIdx.x == 0) report(status, FOCUS_ERR_CAPACITY);
        return;
    }
    const int32_t row_base = win_off[w] - w0;           // first row of the window in the span tensors
    const bool valid1 = a0 + BM < Tw;
    const int n_kv0 = LOCAL ? n_ring + n_win0 : n_ring + 2 * cta + 1;
    const int n_kv1 = valid1 ? (LOCAL ? n_ring + n_win : n_ring + 2 * cta + 2) : 0;
    const int n_kv_max = valid1 ? n_kv1 : n_kv0;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // ---- setup -------------------------------------------------------------
    if (threadIdx.x == 0) {
        mbar_init(smem_addr(&bars->q), 1);
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_addr(&bars->kv_full[s]), 1);
            mbar_init(smem_addr(&bars->kv_empty[s]), 1);
        }
        for (int t = 0; t < 2; ++t) {
            mbar_init(smem_addr(&bars->s_full[t]), 1);
            mbar_init(smem_addr(&bars->p_full[t]), BM);
            mbar_init(smem_addr(&bars->o_full[t]), 1);
        }
        mbar_init(smem_addr(&bars->drain), 1);
        mbar_init(smem_addr(&bars->q_rot), 256);
        mbar_init(smem_addr(&bars->k_rot[0]), 1);
        mbar_init(smem_addr(&bars->k_rot[1]), 1);
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

    if (warp < 4) {
    if constexpr (!ROPE) setmaxnreg_dec<kRegsIssue<D>>();
    if (warp == 0) {
        // ================================================= TMA producer
        if (lane == 0) {
            prefetch_tmap(&tm_q);
            prefetch_tmap(&tm_k);
            prefetch_tmap(&tm_v);
            prefetch_tmap(&tm_rk);
            prefetch_tmap(&tm_rv);
            const uint32_t bq = smem_addr(&bars->q);
            mbar_expect_tx(bq, 2 * C::kTileBytes);
            for (int t = 0; t < 2; ++t)
                load_tile<D>(smem_addr(smem + C::kQOff + t * C::kTileBytes), &tm_q, row_base + a0 + t * BM,
                             GQA ? bh * q_per_kv + member : bh, bq);
            // group g = {V_{g-1}, K_g}: everything MMA iteration g reads, in stage g % 2
            int issued = 0;
            for (int g = 0; g <= n_kv_max && !aborted(bars); ++g) {
                const int st = g & 1, use = g >> 1;
                if (use > 0 && !mbar_wait(smem_addr(&bars->kv_empty[st]), (use - 1) & 1, kWaitNs)) {
                    fail(bars, status);
                    break;
                }
                const uint32_t bf = smem_addr(&bars->kv_full[st]);
                mbar_expect_tx(bf, (uint32_t)(((g >= 1) + (g < n_kv_max)) * C::kTileBytes));
                const uint32_t sbase = smem_addr(smem + C::kSlotOff + 2 * st * C::kTileBytes);
                if (g >= 1) {
                    const int jv = g - 1;
                    const bool ring = jv < n_ring;
                    const int32_t row = ring ? ring_lo + jv * BN : row_base + win_lo + (jv - n_ring) * BN;
                    load_tile<D>(sbase, ring ? &tm_rv : &tm_v, row, bh, bf);
                }
                if (g < n_kv_max) {
                    const bool ring = g < n_ring;
                    const int32_t row = ring ? ring_lo + g * BN : row_base + win_lo + (g - n_ring) * BN;
                    load_tile<D>(sbase + C::kTileBytes, ring ? &tm_rk : &tm_k, row, bh, bf);
                }
                issued = g + 1;
            }
            // drain: every issued copy must land before the CTA can exit
            mbar_wait(smem_addr(&bars->q), 0, kWaitNs);
            for (int g = (issued > 2 ? issued - 2 : 0); g < issued; ++g)
                mbar_wait(smem_addr(&bars->kv_full[g & 1]), (g >> 1) & 1, kWaitNs);
        }
    } else if (warp == 1) {
        // ================================================= MMA issuer
        if (lane == 0) {
            const uint32_t sq = smem_addr(smem + C::kQOff);
            const uint32_t sslot = smem_addr(smem + C::kSlotOff);
            bool ok = mbar_wait(smem_addr(ROPE ? &bars->q_rot : &bars->q), 0, kWaitNs);
            if (!ok) fail(bars, status);
            for (int j = 0; ok && j <= n_kv_max; ++j) {
                const int st = j & 1;
                // K_j of a rotary variant is ready once warps 2-3 have rotated it
                // (they waited for the stage); V alone (the last group) on the stage
                const uint32_t bar = (ROPE && j < n_kv_max) ? smem_addr(&bars->k_rot[st]) : smem_addr(&bars->kv_full[st]);
                if (!mbar_wait(bar, (j >> 1) & 1, kWaitNs)) { ok = false; break; }
                if (ROPE && j < n_kv_max && j >= 1 &&
                    !mbar_wait(smem_addr(&bars->kv_full[st]), (j >> 1) & 1, kWaitNs)) { ok = false; break; }
                const uint32_t vbase = sslot + 2 * st * C::kTileBytes, kbase = vbase + C::kTileBytes;
                tc_fence_after();
                for (int t = 0; t < 2; ++t) {
                    const int nkt = t == 0 ? n_kv0 : n_kv1;
                    if (j >= 1 && j - 1 < nkt) {              // O_t += P_t(j-1) V_{j-1}
                        if (!mbar_wait(smem_addr(&bars->p_full[t]), (j - 1) & 1, kWaitNs)) { ok = false; break; }
                        tc_fence_after();
                        issue_pv<D>(tmem + 256 + t * D, tmem + t * 128, vbase, j - 1 > 0);
                        if (j - 1 == nkt - 1) mma_commit(smem_addr(&bars->o_full[t]));
                    }
                    if (j < nkt) {                           // S_t = Q_t K_j^T
                        issue_qk<D>(tmem + t * 128, sq + t * C::kTileBytes, kbase);
                        mma_commit(smem_addr(&bars->s_full[t]));
                    }
                }
                if (!ok) break;
                mma_commit(smem_addr(&bars->kv_empty[st]));
            }
            if (!ok) fail(bars, status);
            // drain: all issued MMAs complete before TMEM is freed
            mma_commit(smem_addr(&bars->drain));
            mbar_wait(smem_addr(&bars->drain), 0, kWaitNs);
        }
    } else if (ROPE) {
        // ================================================= K rotation (warps 2-3)
        if constexpr (ROPE) {
            constexpr int HALF = D / 16, G = 64 / HALF;
            const int tau = threadIdx.x - 64;
            float2* kb = reinterpret_cast<float2*>(smem + C::kRopeOff) + 4 * 64;
            const int jj = tau % HALF, g = tau / HALF;
            float2 off[8];
            Rot8 step;
            rope_offsets(rope.t.theta, 8 * jj, g, G, off, step);
            const double theta_own = tau < D / 2 ? rope.t.theta[tau] : 0.0;
            for (int j = 0; j < n_kv_max; ++j) {
                const int st = j & 1, slot = 2 * st + 1;        // K_j: stage j % 2, second slot
                if (!mbar_wait(smem_addr(&bars->kv_full[st]), (j >> 1) & 1, kWaitNs)) {
                    fail(bars, status);
                    break;
                }
                if (j >= n_ring) {
                    const int64_t pos0 = (int64_t)win_off[w] + win_lo + (int64_t)(j - n_ring) * BN;
                    if (tau < D / 2) kb[tau] = rope_cs((double)pos0 * theta_own);
                    named_bar_sync(3, 64);
                    float2 cs[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) cs[e] = rope_mul(kb[8 * jj + e], off[e]);
                    Rot8 rot = rot8_make(cs);
                    uint8_t* tile = smem + C::kSlotOff + slot * C::kTileBytes;
                    const int clo = 8 * jj, chi = 8 * jj + D / 2;
#pragma unroll 2
                    for (int m = 0; m < BN / G; ++m) {
                        const int r = g + G * m;
                        uint4* plo = reinterpret_cast<uint4*>(tile + (clo / 64) * kBoxBytes + r * 128 +
                                                              ((((clo % 64) / 8) ^ (r & 7)) << 4));
                        uint4* phi = reinterpret_cast<uint4*>(tile + (chi / 64) * kBoxBytes + r * 128 +
                                                              ((((chi % 64) / 8) ^ (r & 7)) << 4));
                        uint4 lo = *plo, hi = *phi;
                        rot8_apply(lo, hi, rot);
                        *plo = lo;
                        *phi = hi;
                        rot8_step(rot, step);
                    }
                    fence_proxy_async_smem();
                    named_bar_sync(3, 64);
                }
                if (tau == 0) mbar_arrive(smem_addr(&bars->k_rot[st]));
            }
        }
    }
    } else {
        // ================================================= softmax / epilogue
        if constexpr (!ROPE) setmaxnreg_inc<kRegsSoftmax<D>>();
        const int t = (warp - 4) >> 2;                    // 0: warps 4-7, 1: warps 8-11
        const int quarter = warp & 3;                     // TMEM lanes this warp may access
        const int r = quarter * 32 + lane;                // row within the Q tile
        const int32_t aq = a0 + t * BM + r;               // in-window row
        const int n_kv = t == 0 ? n_kv0 : n_kv1;
        const int qt = 2 * cta + t;                       // q-tile index within the window
        const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
        const uint32_t s_addr = tmem + lane_addr + t * 128;
        const uint32_t o_addr = tmem + lane_addr + 256 + t * D;
        // LOCAL: the row's k-mer starts at in-window row lo_row; it sees ring keys
        // [ring_lo, ring_lo + ring_lim) (boundary + earlier in-window FOCUS rows)
        const int32_t c_row = LOCAL ? aq / kdiv : 0;
        const int32_t lo_row = c_row * kdiv;
        const int32_t ring_lim = c_row + bnd;
        float m_run = -INFINITY, l_run = 0.f;
        bool ok = true;
        if constexpr (ROPE) {
            // rotate both Q tiles: thread tau owns pair chunk jj of rows 64 seg + g + G m
            constexpr int HALF = D / 16, G = 64 / HALF;
            const int tau = threadIdx.x - 128, seg = tau >> 6;
            float2* qb = reinterpret_cast<float2*>(smem + C::kRopeOff);    // [4][64]
            const int64_t pos0 = (int64_t)win_off[w] + a0 + 64 * seg;
            if ((tau & 63) < D / 2) qb[seg * 64 + (tau & 63)] = rope_cs((double)pos0 * rope.t.theta[tau & 63]);
            const int jj = tau % HALF, g = (tau / HALF) % G;
            float2 off[8];
            Rot8 step;
            rope_offsets(rope.t.theta, 8 * jj, g, G, off, step);
            named_bar_sync(2, 256);
            float2 cs[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) cs[e] = rope_mul(qb[seg * 64 + 8 * jj + e], off[e]);
            Rot8 rot = rot8_make(cs);
            ok = mbar_wait(smem_addr(&bars->q), 0, kWaitNs);
            if (ok) {
                const int clo = 8 * jj, chi = 8 * jj + D / 2;
#pragma unroll 2
                for (int m = 0; m < 64 / G; ++m) {
                    const int rho = 64 * seg + g + G * m, tq = rho >> 7, rr = rho & 127;
                    uint8_t* tile = smem + C::kQOff + tq * C::kTileBytes;
                    uint4* plo = reinterpret_cast<uint4*>(tile + (clo / 64) * kBoxBytes + rr * 128 +
                                                          ((((clo % 64) / 8) ^ (rr & 7)) << 4));
                    uint4* phi = reinterpret_cast<uint4*>(tile + (chi / 64) * kBoxBytes + rr * 128 +
                                                          ((((chi % 64) / 8) ^ (rr & 7)) << 4));
                    uint4 lo = *plo, hi = *phi;
                    rot8_apply(lo, hi, rot);
                    *plo = lo;
                    *phi = hi;
                    rot8_step(rot, step);
                }
                fence_proxy_async_smem();
            } else {
                fail(bars, status);
            }
            mbar_arrive(smem_addr(&bars->q_rot));
        }
        for (int j = 0; j < n_kv; ++j) {
            if (!mbar_wait(smem_addr(&bars->s_full[t]), j & 1, kWaitNs)) { ok = false; break; }
            tc_fence_after();
            uint32_t sr[128];
            if constexpr (ROPE) {
                tmem_ld32(s_addr + 0, sr);
                tmem_ld32(s_addr + 32, sr + 32);
                tmem_ld32(s_addr + 64, sr + 64);
                tmem_ld32(s_addr + 96, sr + 96);
            } else {
                tmem_ld128(s_addr, sr);
            }
            tmem_wait_ld();
            float* s = reinterpret_cast<float*>(sr);
            // analytic mask
            const bool ring = j < n_ring;
            if (LOCAL) {                                  // visible keys of this tile: columns [lo, hi]
                int32_t lo, hi;
                if (ring) {
                    lo = 0;
                    hi = ring_lim - j * BN - 1;
                } else {
                    const int32_t base = win_lo + (j - n_ring) * BN;
                    lo = lo_row - base;
                    hi = aq - base;
                }
                if (lo > 0 || hi < BN - 1) {
#pragma unroll
                    for (int c = 0; c < BN; ++c)
                        if (c < lo || c > hi) s[c] = -INFINITY;
                }
            } else if (ring) {
                const int lim = Rw - j * BN;              // keys [0, lim) of this tile are visible
                if (lim < BN) {
#pragma unroll
                    for (int c = 0; c < BN; ++c)
                        if (c >= lim) s[c] = -INFINITY;
                }
            } else if (j - n_ring == qt) {                // diagonal tile: key c visible iff c <= r
#pragma unroll
                for (int c = 0; c < BN; ++c)
                    if (c > r) s[c] = -INFINITY;
            }
            // LOCAL rows can meet tiles with no visible key before their first one
            softmax_tile<D, LOCAL>(s, s_addr, o_addr, scale_log2, m_run, l_run, j > 0);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(smem_addr(&bars->p_full[t]));
        }
        // ---- epilogue: O / l -> bf16, staged in this tile's Q buffer ------------
        if (ok && n_kv > 0) ok = mbar_wait(smem_addr(&bars->o_full[t]), 0, kWaitNs);
        if (!ok && n_kv > 0) fail(bars, status);
        __syncwarp();
        if (ok && n_kv > 0) {
            tc_fence_after();
            const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
            uint8_t* stage = smem + C::kQOff + t * C::kTileBytes;     // rows [r] of 2*D bytes, 16-B chunks swizzled
            constexpr int CH = D / 8;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t orr[32];
                tmem_ld32(o_addr + c * 32, orr);
                tmem_wait_ld();
                const uint64_t il2 = f2_pack(inv_l, inv_l);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {          // 4 chunks of 8 values, scaled in pairs
                    uint32_t w4[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        float lo, hi;
                        f2_unpack(f2_mul(f2_pack(__uint_as_float(orr[q4 * 8 + 2 * e]),
                                                 __uint_as_float(orr[q4 * 8 + 2 * e + 1])), il2), lo, hi);
                        w4[e] = pack_bf16x2(lo, hi);
                    }
                    const int chunk = c * 4 + q4;
                    *reinterpret_cast<uint4*>(stage + r * (2 * D) + ((chunk ^ (r & 7)) << 4)) =
                        make_uint4(w4[0], w4[1], w4[2], w4[3]);
                }
            }
            const int32_t bhq = GQA ? query_head_row(H, q_per_kv) : bh;   // Q, O and LSE rows
            if (lse && aq < Tw)
                lse[(int64_t)bhq * T_span + row_base + aq] = (m_run + __log2f(l_run)) * 0.69314718055994531f;
            __syncwarp();
            // the warp stores the 32 rows it staged: 32/CH rows per instruction, coalesced
            __nv_bfloat16* ob = o + ((int64_t)bhq * T_span + row_base + a0 + t * BM) * D;
            constexpr int RPI = 32 / CH;                  // rows per store instruction
            for (int i = 0; i < 32; i += RPI) {
                const int rr = quarter * 32 + i + lane / CH;
                const int chunk = lane % CH;
                if (a0 + t * BM + rr < Tw)
                    *reinterpret_cast<uint4*>(ob + (int64_t)rr * D + chunk * 8) =
                        *reinterpret_cast<const uint4*>(stage + rr * (2 * D) + ((chunk ^ (rr & 7)) << 4));
            }
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

template <int D, bool LOCAL, bool ROPE, bool GQA>
cudaError_t launch_d(const focus_cache& c, const focus_prefill_args& a, int32_t* status, cudaStream_t stream) {
    const int64_t BH = (int64_t)c.B * c.H;
    const int32_t g = c.q_per_kv > 1 ? c.q_per_kv : 1;
    CUtensorMap tq, tk, tv, trk, trv;
    cudaError_t e;
    if ((e = make_map(&tq, a.q, D, a.T_span, BH * g)) != cudaSuccess) return e;
    if ((e = make_map(&tk, a.k, D, a.T_span, BH)) != cudaSuccess) return e;
    if ((e = make_map(&tv, a.v, D, a.T_span, BH)) != cudaSuccess) return e;
    if (c.C_ring > 0) {
        if ((e = make_map(&trk, c.ring_k, D, c.C_ring, BH)) != cudaSuccess) return e;
        if ((e = make_map(&trv, c.ring_v, D, c.C_ring, BH)) != cudaSuccess) return e;
    } else {                                   // no ring: the maps are never read
        trk = tk;
        trv = tv;
    }
    const int smem = Cfg<D>::kSmem;
    e = cudaFuncSetAttribute(prefill_tc_kernel<D, LOCAL, ROPE, GQA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem);
    if (e != cudaSuccess) return e;
    if constexpr (!ROPE) {
        // the register split needs the launch registers it was sized for: with
        // fewer, the softmax warpgroups' setmaxnreg.inc could never be served
        cudaFuncAttributes fa;
        if ((e = cudaFuncGetAttributes(&fa, prefill_tc_kernel<D, LOCAL, ROPE, GQA>)) != cudaSuccess) return e;
        if (fa.numRegs < kLaunchRegs) return cudaErrorInvalidConfiguration;
    }
    const int ctas_pw = (a.max_rows + 2 * BM - 1) / (2 * BM);
    dim3 grid((unsigned)((a.w_end - a.w_begin) * ctas_pw * g), c.H, c.B);
    RopeArg<ROPE> rope;
    if constexpr (ROPE) rope_table_fill(&rope.t, D, c.rope_theta);
    else rope.unused = 0;
    prefill_tc_kernel<D, LOCAL, ROPE, GQA><<<grid, kThreads, smem, stream>>>(
        tq, tk, tv, trk, trv, (__nv_bfloat16*)a.o, a.lse, a.T_span, a.d_win_off, a.d_ring_off,
        a.w_begin, a.w_end, ctas_pw, c.H, c.C_ring, a.scale * 1.4426950408889634f, status, c.k_per_window, rope, g);
    return cudaGetLastError();
}

}  // namespace

template <bool GQA>
cudaError_t dispatch(const focus_cache& c, const focus_prefill_args& a, int32_t* status, cudaStream_t stream,
                     bool local, bool rope) {
    if (c.d == 128) {
        if (rope) return local ? launch_d<128, true, true, GQA>(c, a, status, stream)
                               : launch_d<128, false, true, GQA>(c, a, status, stream);
        return local ? launch_d<128, true, false, GQA>(c, a, status, stream)
                     : launch_d<128, false, false, GQA>(c, a, status, stream);
    }
    if (rope) return local ? launch_d<64, true, true, GQA>(c, a, status, stream)
                           : launch_d<64, false, true, GQA>(c, a, status, stream);
    return local ? launch_d<64, true, false, GQA>(c, a, status, stream)
                 : launch_d<64, false, false, GQA>(c, a, status, stream);
}

// Work items of at most kPersistentMaxRows / 128 K/V tiles (ring capacity plus the
// longest window) spend a large share of their time in per-CTA start-up and the O
// epilogue; the persistent kernel overlaps those with the neighbouring items.
// Longer items keep one CTA per item: the hardware's block scheduling balances
// them better, and that kernel's per-tile loop is ~4% faster.
constexpr int64_t kPersistentMaxRows = 4096;

bool prefill_persistent_case(const focus_cache& c, const focus_prefill_args& a) {
    const bool local = (a.flags & FOCUS_PREFILL_KMER_LOCAL) != 0;
    // the persistent kernel numbers its work items with 32-bit arithmetic
    const int64_t g = c.q_per_kv > 1 ? c.q_per_kv : 1;
    const int64_t items = (int64_t)(a.w_end - a.w_begin) * ((a.max_rows + 2 * BM - 1) / (2 * BM)) * g * c.H * c.B;
    return !(a.flags & FOCUS_PREFILL_LEGACY_MMA) && !local && (int64_t)c.C_ring + a.max_rows <= kPersistentMaxRows &&
           items <= INT32_MAX;
}

namespace {

// The rotary embedding with a workspace for the rotated q and k (one layout for
// both uses: the persistent kernel's per-head counters, then the rotated q and k):
// - grouped-query heads on short work items: the persistent kernel rotates q and
//   k into it itself, beside the attention (the g query heads of a K/V head share
//   every angle, and there are fewer K rows to rotate, so the rotation keeps ahead
//   of the attention: 128 kb with g = 2, 2.34 ms against 2.61 ms with the pass);
// - otherwise a pass rotates them there first and the attention runs as without
//   the embedding (128 kb with g = 1: 2.79 ms against 2.99 ms with the rotation
//   inside the persistent kernel);
// except for the k-mer-tiled kernel, which rotates its tiles in place and needs no
// workspace. Without the workspace, the one-CTA-per-item kernel rotates the
// tiles each CTA loads.
constexpr int32_t kRopeFusedMinGroup = 2;

bool rope_workspace_ok(const focus_cache& c, const focus_prefill_args& a) {
    if (!(c.rope_theta > 0.f) || (a.flags & FOCUS_PREFILL_LEGACY_MMA)) return false;
    return a.workspace && a.workspace_bytes >= prefill::persistent_workspace_bytes(c, a);
}

bool rope_fused(const focus_cache& c, const focus_prefill_args& a) {
    return rope_workspace_ok(c, a) && c.q_per_kv >= kRopeFusedMinGroup && prefill_persistent_case(c, a);
}

// The k-mer-tiled kernel (which rotates q and k in place itself: it reads each
// window row in one work item per query head).
bool kmer_case(const focus_cache& c, const focus_prefill_args& a) {
    int32_t RB, tiles;
    return !(a.flags & FOCUS_PREFILL_LEGACY_MMA) && (a.flags & FOCUS_PREFILL_KMER_LOCAL) &&
           prefill::kmer_tiling(c, a, &RB, &tiles);
}

bool rope_pass(const focus_cache& c, const focus_prefill_args& a) {
    return rope_workspace_ok(c, a) && !rope_fused(c, a) && !kmer_case(c, a);
}

int32_t prefill_kernel_choice_plain(const focus_cache& c, const focus_prefill_args& a) {
    if (a.flags & FOCUS_PREFILL_LEGACY_MMA) return FOCUS_PREFILL_KERNEL_LEGACY;
    const bool rope = c.rope_theta > 0.f;
    if (kmer_case(c, a)) return FOCUS_PREFILL_KERNEL_KMER;
    if ((!rope || rope_fused(c, a)) && prefill_persistent_case(c, a)) return FOCUS_PREFILL_KERNEL_PERSISTENT;
    return FOCUS_PREFILL_KERNEL_PER_ITEM;
}

}  // namespace

int32_t prefill_kernel_choice(const focus_cache& c, const focus_prefill_args& a) {
    if (rope_pass(c, a)) {
        focus_cache c0 = c;
        c0.rope_theta = 0.f;
        return prefill_kernel_choice_plain(c0, a) | FOCUS_PREFILL_KERNEL_ROTATION_PASS;
    }
    return prefill_kernel_choice_plain(c, a);
}

size_t prefill_workspace_bytes(const focus_cache& c, const focus_prefill_args& a) {
    return (a.flags & FOCUS_PREFILL_LEGACY_MMA) || kmer_case(c, a) ? 0 : prefill::persistent_workspace_bytes(c, a);
}

namespace {

cudaError_t launch_plain(const focus_cache& c, const focus_prefill_args& a, int32_t* status, cudaStream_t stream) {
    const bool local = (a.flags & FOCUS_PREFILL_KMER_LOCAL) != 0, rope = c.rope_theta > 0.f;
    const int32_t kernel = prefill_kernel_choice_plain(c, a);
    if (kernel == FOCUS_PREFILL_KERNEL_PERSISTENT) return prefill::launch_prefill_tc_persistent(c, a, status, stream);
    if (kernel == FOCUS_PREFILL_KERNEL_KMER) return prefill::launch_prefill_tc_kmer(c, a, status, stream);
    if (c.q_per_kv > 1) return dispatch<true>(c, a, status, stream, local, rope);
    return dispatch<false>(c, a, status, stream, local, rope);
}

}  // namespace

cudaError_t launch_prefill_tc(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                              cudaStream_t stream) {
    if (rope_pass(c, a)) {
        // q rows, then k rows, after the counters; the attention reads those
        const int64_t g = c.q_per_kv > 1 ? c.q_per_kv : 1;
        char* q_rot = static_cast<char*>(a.workspace) + prefill::rope_counter_bytes(c);
        char* k_rot = q_rot + (size_t)c.B * c.H * g * (size_t)a.T_span * c.d * 2;
        cudaError_t e = prefill::launch_rope_rotate(c, a, q_rot, k_rot, stream);
        if (e != cudaSuccess) return e;
        focus_cache c0 = c;
        c0.rope_theta = 0.f;
        focus_prefill_args a0 = a;
        a0.q = q_rot;
        a0.k = k_rot;
        return launch_plain(c0, a0, status, stream);
    }
    return launch_plain(c, a, status, stream);
}

}  // namespace focus
