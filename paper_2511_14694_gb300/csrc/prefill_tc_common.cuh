// Shared by the two tcgen05 prefill kernels: prefill_tc.cu (one CTA per work
// item of two 128-row Q tiles; every mask and the rotary embedding) and
// prefill_tc_persistent.cu (one CTA per SM walking the work items; appendix
// mask only). Tile geometry, shared-memory layout, barriers, the online softmax
// of one S tile, and the TMA tensor maps.
#pragma once

#include <cudaTypedefs.h>

#include "common.cuh"
#include "sm100.cuh"

namespace focus {
namespace prefill {

using namespace sm100;

constexpr int BM = 128;             // rows per Q tile
constexpr int BN = 128;             // keys per K/V tile
constexpr int kStages = 2;          // K/V stages, each one MMA iteration's {V_{j-1}, K_j}
constexpr int kSlots = 2 * kStages; // K/V tiles in shared memory (stage s: slots 2s (V) and 2s + 1 (K))
constexpr int kThreads = 384;       // 12 warps
constexpr int kLaunchRegs = 168;    // registers per thread at launch: 65,536 / 384 rounded down to 8
constexpr int kBoxBytes = 128 * 128;   // one TMA box: 128 rows x 64 bf16 (128 B, swizzled)
constexpr uint64_t kWaitNs = 2000000000ull;   // 2 s bound on any wait
constexpr float kRescaleThreshold = 8.0f;     // log2 units: rescale O only if the max grows by > 2^8

// Shared scratch of one 64-thread group rotating q/k rows in the persistent
// kernel: 64 unit start angles and 64 x 8 row offsets (float2).
constexpr int kRopeGroupScratch = 64 * 8 + 64 * 8 * 8;

template <int D>
struct Cfg {
    static constexpr int kBoxes = D / 64;                       // TMA boxes per 128-row tile
    static constexpr int kTileBytes = kBoxes * kBoxBytes;       // one Q/K/V tile
    static constexpr int kQOff = 0;
    static constexpr int kSlotOff = 2 * kTileBytes;
    static constexpr int kBarOff = kSlotOff + kSlots * kTileBytes;
    static constexpr int kRopeOff = kBarOff + 256;              // float2 [4][64] Q bases + [64] K bases
    static constexpr int kSmem = kRopeOff + 5 * 64 * 8 + 1024;  // + alignment slack
    // persistent kernel: no rotary bases; O staging of 8 warps x 32 rows x 64 B
    static constexpr int kStageOff = kBarOff + 256;
    static constexpr int kSmemPersistent = kStageOff + 8 * 2048 + 1024;
    // persistent kernel with the rotary embedding: one rotating group's scratch
    static constexpr int kRopeScratchOff = kStageOff + 8 * 2048;
    static constexpr int kSmemPersistentRope = kRopeScratchOff + kRopeGroupScratch + 1024;
};

struct Bars {
    uint64_t q;
    uint64_t kv_full[kStages];   // stage landed (TMA complete_tx)
    uint64_t kv_empty[kStages];  // the stage's MMAs have completed
    uint64_t s_full[2];
    uint64_t p_full[2];
    uint64_t o_full[2];
    uint64_t drain;
    uint64_t q_rot;       // rotary embedding: the Q tiles are rotated
    uint64_t k_rot[kStages];  // rotary embedding: the K tile of the stage is rotated
    uint64_t o_free[2];   // persistent: the epilogue has read O_t
    uint64_t q_free;      // persistent: every QK of the current item has completed, Q may be reloaded
    uint32_t tmem;
    int32_t abort;
};
static_assert(sizeof(Bars) <= 256, "barriers must fit their 256-byte slot");

__device__ __forceinline__ void fail(Bars* bars, int32_t* status) {
    report(status, FOCUS_ERR_TIMEOUT);
    atomicExch(&bars->abort, 1);
}
__device__ __forceinline__ bool aborted(Bars* bars) { return *(volatile int32_t*)&bars->abort != 0; }

// One 128-row tile of a [BH][rows][D] bf16 tensor into shared memory as D/64 TMA
// boxes of 128 rows x 64 columns (128-byte swizzle), completing on `bar`.
template <int D>
__device__ __forceinline__ void load_tile(uint32_t dst, const CUtensorMap* map, int32_t row, int32_t bh, uint32_t bar) {
#pragma unroll
    for (int x = 0; x < D / 64; ++x) tma_load_3d(dst + x * kBoxBytes, map, x * 64, row, bh, bar);
}

// S (TMEM, 128 fp32 columns) = Q K^T for one 128-row Q tile and one 128-key K
// tile, both K-major in shared memory: D/16 MMAs of 128x128x16.
template <int D>
__device__ __forceinline__ void issue_qk(uint32_t s_tmem, uint32_t qbase, uint32_t kbase) {
    constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, false, false);
    // the start address is the descriptor's low field (address >> 4, shared
    // addresses < 256 KB), so an offset is added to a base descriptor
    const uint64_t dq = smem_desc_sw128(qbase, 16, 1024), dk = smem_desc_sw128(kbase, 16, 1024);
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = ((kk / 4) * kBoxBytes + (kk % 4) * 32) >> 4;
        mma_ss(s_tmem, dq + off, dk + off, idesc, kk > 0 ? 1u : 0u);
    }
}

// O (TMEM, D fp32 columns) (+)= P V for one Q tile: P bf16 in TMEM over S, V an
// MN-major 128-key tile in shared memory; BN/16 MMAs of 128xDx16. `accumulate` is
// false for the first tile of an item, whose PV overwrites O.
template <int D>
__device__ __forceinline__ void issue_pv(uint32_t o_tmem, uint32_t p_tmem, uint32_t vbase, bool accumulate) {
    constexpr uint32_t idesc = idesc_bf16_f32(BM, D, false, true);
    const uint64_t dv = smem_desc_sw128(vbase, kBoxBytes, 1024);
#pragma unroll
    for (int kk = 0; kk < BN / 16; ++kk)
        mma_ts(o_tmem, p_tmem + kk * 8, dv + (uint64_t)(kk * 2048 >> 4), idesc, (accumulate || kk > 0) ? 1u : 0u);
}

// Online softmax of one S tile in the log2 domain for the row this thread owns:
// s holds the row's BN masked scores, (m_run, l_run) the running max and sum.
// P = 2^(s scale - m) goes back to TMEM over S as bf16 pairs (two 32-column
// stores); when the max grows by more than 2^kRescaleThreshold for any row of the
// warp, l and, once a PV has written it (has_o), O_t in TMEM are rescaled.
// ZERO_FLOOR: a row whose scores have all been -inf so far subtracts 0 instead of
// -inf, so that every p is exactly 0 (masks that can hide a whole tile of a row).
template <int D, bool ZERO_FLOOR>
__device__ __forceinline__ void softmax_tile(const float* s, uint32_t s_addr, uint32_t o_addr, float scale_log2,
                                             float& m_run, float& l_run, bool has_o) {
    // row max: four independent chains of three-input max (depth 16, not 128)
    float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
    for (int c = 0; c < BN; c += 8) {
        mx[0] = max3f(mx[0], s[c + 0], s[c + 1]);
        mx[1] = max3f(mx[1], s[c + 2], s[c + 3]);
        mx[2] = max3f(mx[2], s[c + 4], s[c + 5]);
        mx[3] = max3f(mx[3], s[c + 6], s[c + 7]);
    }
    const float mt = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
    const float m_new = fmaxf(m_run, mt * scale_log2);
    const bool need = m_new > m_run + kRescaleThreshold;
    const bool any_need = __any_sync(0xffffffffu, need);
    const float factor = need ? ex2_approx(m_run - m_new) : 1.f;
    if (need) m_run = m_new;
    l_run *= factor;
    // p = 2^(s * scale_log2 - m): packed FMA on pairs, ex2 per element, row sum in
    // four packed partial sums (independent chains)
    const float m_sub = (ZERO_FLOOR && m_run == -INFINITY) ? 0.f : m_run;
    const uint64_t sc2 = f2_pack(scale_log2, scale_log2), nm2 = f2_pack(-m_sub, -m_sub);
    uint64_t acc2[4] = {0, 0, 0, 0};
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
        uint32_t pk[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            float x0, x1;
            f2_unpack(f2_fma(f2_pack(s[h2 * 64 + 2 * i], s[h2 * 64 + 2 * i + 1]), sc2, nm2), x0, x1);
            const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
            acc2[i & 3] = f2_add(acc2[i & 3], f2_pack(p0, p1));
            pk[i] = pack_bf16x2(p0, p1);
        }
        tmem_st32(s_addr + h2 * 32, pk);
    }
    float lsum = 0.f;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        float lo, hi;
        f2_unpack(acc2[a], lo, hi);
        lsum += lo + hi;
    }
    l_run += lsum;
    // Lazy rescale of O_t (written by the previous PV, which completed before this
    // S tile was signalled; the next PV waits for this thread's arrival).
    if (any_need && has_o) {
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
            uint32_t orr[32];
            tmem_ld32(o_addr + c * 32, orr);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) orr[i] = __float_as_uint(__uint_as_float(orr[i]) * factor);
            tmem_st32(o_addr + c * 32, orr);
        }
    }
}

// ---------------------------------------------------------------- rotary embedding

// Kernel argument: the rotary table only for the ROPE variants.
template <bool ROPE>
struct RopeArg {
    RopeTable t;
};
template <>
struct RopeArg<false> {
    int unused;
};

// Rotation of eight column pairs (one 16-byte chunk and its partner d/2 columns
// on), as four packed pairs of element pairs: c = cos, s = sin, n = -sin.
struct Rot8 {
    uint64_t c[4], s[4], n[4];
};

__device__ __forceinline__ Rot8 rot8_make(const float2* cs) {
    Rot8 r;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        r.c[k] = f2_pack(cs[2 * k].x, cs[2 * k + 1].x);
        r.s[k] = f2_pack(cs[2 * k].y, cs[2 * k + 1].y);
        r.n[k] = f2_pack(-cs[2 * k].y, -cs[2 * k + 1].y);
    }
    return r;
}

// y_lo = x_lo c - x_hi s, y_hi = x_hi c + x_lo s on bf16 chunks, rounded once to bf16.
__device__ __forceinline__ void rot8_apply(uint4& lo, uint4& hi, const Rot8& r) {
    uint32_t* l = reinterpret_cast<uint32_t*>(&lo);
    uint32_t* h = reinterpret_cast<uint32_t*>(&hi);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint64_t xl = f2_pack(__uint_as_float(l[k] << 16), __uint_as_float(l[k] & 0xffff0000u));
        const uint64_t xh = f2_pack(__uint_as_float(h[k] << 16), __uint_as_float(h[k] & 0xffff0000u));
        const uint64_t yl = f2_fma(xh, r.n[k], f2_mul(xl, r.c[k]));
        const uint64_t yh = f2_fma(xl, r.s[k], f2_mul(xh, r.c[k]));
        float a, b;
        f2_unpack(yl, a, b);
        l[k] = pack_bf16x2(a, b);
        f2_unpack(yh, a, b);
        h[k] = pack_bf16x2(a, b);
    }
}

// r <- r turned further by the angles of st.
__device__ __forceinline__ void rot8_step(Rot8& r, const Rot8& st) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint64_t c = f2_fma(r.c[k], st.c[k], f2_mul(r.s[k], st.n[k]));
        const uint64_t sn = f2_fma(r.s[k], st.c[k], f2_mul(r.c[k], st.s[k]));
        const uint64_t n = f2_fma(r.n[k], st.c[k], f2_mul(r.c[k], st.n[k]));
        r.c[k] = c;
        r.s[k] = sn;
        r.n[k] = n;
    }
}

// (cos, sin) of the small angles g theta_i and G theta_i (|angle| <= 16) for the
// eight pairs i0..i0+7: fp32 is accurate to ~1e-6 rad here.
__device__ __forceinline__ void rope_offsets(const double* theta, int i0, int g, int G, float2* off, Rot8& step) {
    float2 st[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float th = (float)theta[i0 + e];
        __sincosf((float)g * th, &off[e].y, &off[e].x);
        __sincosf((float)G * th, &st[e].y, &st[e].x);
    }
    step = rot8_make(st);
}

// 3-D map over a [BH][rows][d] bf16 tensor, box = box_rows rows x 64 columns
// (a multiple of 8, <= 128; a tile's 128 rows by default), 128-byte swizzle.
cudaError_t make_map(CUtensorMap* m, const void* ptr, int d, int64_t rows, int64_t bh, int box_rows = 128);

// The persistent kernel (appendix mask). With the rotary embedding (grouped-query
// heads) it rotates Q and K itself, into the caller's workspace
// (persistent_workspace_bytes).
cudaError_t launch_prefill_tc_persistent(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                                         cudaStream_t stream);
// The k-mer-local kernel with query tiles cut at k-mer boundaries
// (prefill_tc_kmer.cu): whether the span qualifies (needs args.h_k_per_window),
// and then its ring rows per tile (RB) and tiles per window.
bool kmer_tiling(const focus_cache& c, const focus_prefill_args& a, int32_t* RB, int32_t* max_tiles);
cudaError_t launch_prefill_tc_kmer(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                                   cudaStream_t stream);

// Workspace bytes for the rotary embedding (the persistent kernel's own rotation
// and the pass share the layout): 0 without it; with it a 256-byte block of
// per-head counters, then Q and K of the span, rotated.
size_t persistent_workspace_bytes(const focus_cache& c, const focus_prefill_args& a);

// Bytes of the per-head counters at the start of that workspace.
size_t rope_counter_bytes(const focus_cache& c);

// The rotary embedding as a pass before the attention (rope.cu): writes the span's
// rotated q rows to q_rot ([B][H g][T_span][d] bf16) and its k rows to k_rot
// ([B][H][T_span][d]).
cudaError_t launch_rope_rotate(const focus_cache& c, const focus_prefill_args& a, void* q_rot, void* k_rot,
                               cudaStream_t stream);

}  // namespace prefill
}  // namespace focus
