// Single-token decode against the compressed KV cache (App. A.2, streaming
// inference: the retained FOCUS K/V of earlier windows are the history, the
// current window's rows are attended causally; the new row sees itself).
//
// HBM-bound: every K/V row of the ring and of the window buffer is read once
// per K/V head (grouped query heads share the pass, see the tensor-core kernel).
// Split-K over keys: grid (split, head, sequence); each CTA streams a chunk of
// keys with 16-byte loads (d/8 lanes per key row, several rows in flight per
// thread), keeps a per-lane-group online softmax in registers, merges the
// groups through shared memory and writes one partial (m, l, o) per split. A
// second small kernel merges the splits with their log-sum-exp weights and
// advances win_fill.
#include <mutex>

#include "common.cuh"
#include "sm100.cuh"

namespace focus {
namespace {

// Fixed scratch for focus_attn_decode_noalloc. Callers that cannot allocate
// device memory get their split-K partials here instead of in a workspace of
// their own. Every device that loads the library keeps these bytes until the
// process exits, and all calls share them.
static __device__ __align__(256) unsigned char g_decode_scratch[FOCUS_DECODE_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxScratchDevices = 64;
void* g_scratch_ptr[kMaxScratchDevices];
std::mutex g_scratch_mu;

constexpr int kDecodeChunk = 1024;   // keys per split
constexpr int kDecodeThreads = 128;  // consumer threads (plus one producer warp)
constexpr int kStages = 4;           // shared-memory stages in flight per CTA
template <int D>
constexpr int kStageRows = 8192 / (2 * D);   // 8 KB of K and 8 KB of V per stage
constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s bound on any wait
template <int D>
constexpr int decode_groups() { return (kDecodeThreads / 32) * (32 / (D / 8)); }   // lane groups per CTA
template <int D, int QG>
constexpr int decode_smem_bytes() {   // K/V stages + full/empty barriers + the group merge buffers (per query)
    return 2 * kStages * kStageRows<D> * D * 2 + 2 * kStages * 8 + QG * (2 * decode_groups<D>() * 4 +
           decode_groups<D>() * D * 4);
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float* f) {
    const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float2 x = __bfloat1622float2(p[i]);
        f[2 * i] = x.x;
        f[2 * i + 1] = x.y;
    }
}

__device__ __forceinline__ bool decode_state_ok(int32_t R, int32_t fill, int32_t widx, const int32_t* ks,
                                                int32_t n_windows, int32_t W, int32_t C_ring, int32_t C_win,
                                                int32_t* Tw_out, const int32_t* W_per_window) {
    if (widx < 0 || widx >= n_windows || R < 0 || R > C_ring) return false;
    const int32_t Tw = (int32_t)window_rows(cache_window_len(W_per_window, W, widx), ks[widx], true);
    *Tw_out = Tw;
    return fill >= 0 && fill < Tw && fill < C_win;
}

// Split kernel: 4 consumer warps + 1 producer warp. The producer streams the
// split's key rows as contiguous bulk copies (ring part, window part, new row)
// into a ring of shared-memory stages; consumers read each row with d/8 lanes
// (16 B each, conflict-free), reduce the dot product with shuffles and keep a
// per-lane-group online softmax (log2 domain) in registers.
//
// Grouped-query heads (q_per_kv = g > 1): one CTA serves QG of the g query
// heads that share its K/V head, so each K/V row it streams is used QG times
// (blockIdx.y = kv head * (g / QG) + which QG-slice of the group). Even groups
// go to the tensor-core kernel below; this one serves g = 1 and odd g (QG = 1).
template <int D, int QG>
__global__ void __launch_bounds__(kDecodeThreads + 32) decode_split_kernel(
        const uint4* __restrict__ ring_k, const uint4* __restrict__ ring_v, uint4* __restrict__ win_k,
        uint4* __restrict__ win_v, const int32_t* __restrict__ ring_len, const int32_t* __restrict__ win_fill,
        const int32_t* __restrict__ win_idx, const int32_t* __restrict__ ks, int32_t n_windows, int32_t W,
        int32_t H, int32_t C_ring, int32_t C_win, const uint4* __restrict__ q, const uint4* __restrict__ k_new,
        const uint4* __restrict__ v_new, float scale_log2, float2* __restrict__ ws_ml, float* __restrict__ ws_o,
        int32_t n_splits, int32_t* status, const int32_t* __restrict__ W_per_window, int32_t q_per_kv) {
    using namespace sm100;
    constexpr int CPR = D / 8;          // 16-byte chunks per row = lanes per key
    constexpr int GPW = 32 / CPR;       // key groups per warp
    constexpr int NG = (kDecodeThreads / 32) * GPW;
    static_assert(NG == decode_groups<D>(), "group count");
    constexpr int CH = kStageRows<D>;   // key rows per stage
    constexpr int ROWB = D * 2;         // bytes per row
    const int slices = q_per_kv / QG;
    const int b = blockIdx.z, h = blockIdx.y / slices, slice = blockIdx.y % slices, split = blockIdx.x;
    const int64_t bh = (int64_t)b * H + h;                         // K/V head
    const int64_t bhq0 = bh * q_per_kv + (int64_t)slice * QG;      // first of this CTA's query heads
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    const int32_t R = ring_len[b], fill = win_fill[b], widx = win_idx[b];
    int32_t Tw = 0;
    const bool state_ok = decode_state_ok(R, fill, widx, ks, n_windows, W, C_ring, C_win, &Tw, W_per_window);
    const int64_t total = (int64_t)R + fill + 1;
    const int64_t s0 = (int64_t)split * kDecodeChunk;
    const int64_t s1 = min(total, s0 + kDecodeChunk);
    if (!state_ok || s0 >= s1) {
        if (!state_ok && split == 0 && blockIdx.y == 0 && tid == 0) report(status, FOCUS_ERR_CAPACITY);
        for (int j = 0; j < QG; ++j) {
            float* wo = ws_o + ((bhq0 + j) * n_splits + split) * D;
            for (int c = tid; c < D; c += blockDim.x) wo[c] = 0.f;
            if (tid == 0) ws_ml[(bhq0 + j) * n_splits + split] = make_float2(-INFINITY, 0.f);
        }
        return;
    }
    if (split == 0 && slice == 0 && tid < CPR) {      // append the new row to the window buffer
        win_k[(bh * C_win + fill) * CPR + tid] = k_new[bh * CPR + tid];
        win_v[(bh * C_win + fill) * CPR + tid] = v_new[bh * CPR + tid];
    }

    extern __shared__ __align__(128) unsigned char smem[];
    uint8_t* sK = smem;                                   // [kStages][CH][D] bf16
    uint8_t* sV = smem + kStages * CH * ROWB;             // [kStages][CH][D] bf16
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + 2 * kStages * CH * ROWB);
    uint64_t* empty = full + kStages;
    float* sm_m = reinterpret_cast<float*>(empty + kStages);   // [QG][NG]
    float* sm_l = sm_m + QG * NG;                               // [QG][NG]
    float* sm_acc = sm_l + QG * NG;                             // [QG][NG][D]
    __shared__ int32_t abort_flag;
    const int n_chunks = (int)((s1 - s0 + CH - 1) / CH);

    if (tid == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(smem_addr(&full[i]), 1);
            mbar_init(smem_addr(&empty[i]), kDecodeThreads / 32);
        }
        abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();

    if (warp == kDecodeThreads / 32) {
        // ------------------------------------------------ producer
        if (lane == 0) {
            const uint8_t* rk = reinterpret_cast<const uint8_t*>(ring_k) + bh * (int64_t)C_ring * ROWB;
            const uint8_t* rv = reinterpret_cast<const uint8_t*>(ring_v) + bh * (int64_t)C_ring * ROWB;
            const uint8_t* wk = reinterpret_cast<const uint8_t*>(win_k) + bh * (int64_t)C_win * ROWB;
            const uint8_t* wv = reinterpret_cast<const uint8_t*>(win_v) + bh * (int64_t)C_win * ROWB;
            const uint8_t* nk = reinterpret_cast<const uint8_t*>(k_new) + bh * ROWB;
            const uint8_t* nv = reinterpret_cast<const uint8_t*>(v_new) + bh * ROWB;
            int issued = 0;
            for (int c = 0; c < n_chunks; ++c) {
                const int st = c % kStages, use = c / kStages;
                if (use > 0 && !mbar_wait(smem_addr(&empty[st]), (use - 1) & 1, kWaitNs)) {
                    report(status, FOCUS_ERR_TIMEOUT);
                    atomicExch(&abort_flag, 1);
                    break;
                }
                const int64_t k0 = s0 + (int64_t)c * CH, k1 = min(s1, k0 + CH);
                const uint32_t bar = smem_addr(&full[st]);
                mbar_expect_tx(bar, (uint32_t)((k1 - k0) * ROWB * 2));
                const uint32_t dk = smem_addr(sK + st * CH * ROWB), dv = smem_addr(sV + st * CH * ROWB);
                int64_t a = k0, e = min(k1, (int64_t)R);               // ring rows
                if (a < e) {
                    bulk_load(dk, rk + a * ROWB, (uint32_t)((e - a) * ROWB), bar);
                    bulk_load(dv, rv + a * ROWB, (uint32_t)((e - a) * ROWB), bar);
                }
                a = max(k0, (int64_t)R);
                e = min(k1, (int64_t)R + fill);                        // current-window rows
                if (a < e) {
                    const uint32_t off = (uint32_t)((a - k0) * ROWB);
                    bulk_load(dk + off, wk + (a - R) * ROWB, (uint32_t)((e - a) * ROWB), bar);
                    bulk_load(dv + off, wv + (a - R) * ROWB, (uint32_t)((e - a) * ROWB), bar);
                }
                if (k1 == total) {                                      // the new row itself
                    const uint32_t off = (uint32_t)((total - 1 - k0) * ROWB);
                    bulk_load(dk + off, nk, ROWB, bar);
                    bulk_load(dv + off, nv, ROWB, bar);
                }
                issued = c + 1;
            }
            for (int c = max(0, issued - kStages); c < issued; ++c)    // drain before exit
                mbar_wait(smem_addr(&full[c % kStages]), (c / kStages) & 1, kWaitNs);
        }
        __syncthreads();
        return;
    }

    // ---------------------------------------------------- consumers
    const int sub = lane % CPR;
    const int grp = warp * GPW + lane / CPR;
    float qf[QG][8];
#pragma unroll
    for (int j = 0; j < QG; ++j) {
        bf16x8_to_f32(q[(bhq0 + j) * CPR + sub], qf[j]);
#pragma unroll
        for (int e = 0; e < 8; ++e) qf[j][e] *= scale_log2;
    }
    float m[QG], l[QG], acc[QG][8];
#pragma unroll
    for (int j = 0; j < QG; ++j) {
        m[j] = -INFINITY;
        l[j] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[j][e] = 0.f;
    }

    for (int c = 0; c < n_chunks; ++c) {
        const int st = c % kStages;
        if (!mbar_wait(smem_addr(&full[st]), (c / kStages) & 1, kWaitNs) || abort_flag) {
            report(status, FOCUS_ERR_TIMEOUT);
            break;
        }
        const int nrow = (int)min((int64_t)CH, s1 - (s0 + (int64_t)c * CH));
        const uint8_t* kb = sK + st * CH * ROWB + sub * 16;
        const uint8_t* vb = sV + st * CH * ROWB + sub * 16;
        constexpr int U = CH / NG;
        float s[QG][U];
        uint4 vr[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int r = grp + u * NG;
            const bool ok = r < nrow;
            const uint4 kr = ok ? *reinterpret_cast<const uint4*>(kb + r * ROWB) : make_uint4(0, 0, 0, 0);
            vr[u] = ok ? *reinterpret_cast<const uint4*>(vb + r * ROWB) : make_uint4(0, 0, 0, 0);
            float kf[8];
            bf16x8_to_f32(kr, kf);
#pragma unroll
            for (int j = 0; j < QG; ++j) {
                float d0 = 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) d0 = fmaf(qf[j][e], kf[e], d0);
                s[j][u] = d0;
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_addr(&empty[st]));     // this warp is done with the stage
#pragma unroll
        for (int off = CPR / 2; off >= 1; off >>= 1) {
#pragma unroll
            for (int j = 0; j < QG; ++j)
#pragma unroll
                for (int u = 0; u < U; ++u) s[j][u] += __shfl_xor_sync(0xffffffffu, s[j][u], off);
        }
#pragma unroll
        for (int j = 0; j < QG; ++j) {
            float mb = -INFINITY;
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (grp + u * NG >= nrow) s[j][u] = -INFINITY;
                mb = fmaxf(mb, s[j][u]);
            }
            const float mn = fmaxf(m[j], mb);
            if (mn == -INFINITY) continue;
            if (mn > m[j]) {
                const float corr = ex2_approx(m[j] - mn);
                l[j] *= corr;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[j][e] *= corr;
                m[j] = mn;
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            float vf[8];
            bf16x8_to_f32(vr[u], vf);
#pragma unroll
            for (int j = 0; j < QG; ++j) {
                if (m[j] == -INFINITY) continue;
                const float p = ex2_approx(s[j][u] - m[j]);
                l[j] += p;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[j][e] = fmaf(p, vf[e], acc[j][e]);
            }
        }
    }

#pragma unroll
    for (int j = 0; j < QG; ++j) {
        if (sub == 0) { sm_m[j * NG + grp] = m[j]; sm_l[j * NG + grp] = l[j]; }
#pragma unroll
        for (int e = 0; e < 8; ++e) sm_acc[(j * NG + grp) * D + sub * 8 + e] = acc[j][e];
    }
    asm volatile("bar.sync 1, %0;" ::"n"(kDecodeThreads));       // consumers only
    for (int col = tid; col < QG * D; col += kDecodeThreads) {
        const int j = col / D, cc = col % D;
        float M = -INFINITY;
#pragma unroll
        for (int g = 0; g < NG; ++g) M = fmaxf(M, sm_m[j * NG + g]);
        float L = 0.f, A = 0.f;
        if (M != -INFINITY) {
#pragma unroll
            for (int g = 0; g < NG; ++g) {
                const float f = ex2_approx(sm_m[j * NG + g] - M);
                L = fmaf(sm_l[j * NG + g], f, L);
                A = fmaf(sm_acc[(j * NG + g) * D + cc], f, A);
            }
        }
        ws_o[((bhq0 + j) * n_splits + split) * D + cc] = A;
        if (cc == 0) ws_ml[(bhq0 + j) * n_splits + split] = make_float2(M, L);
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// Grouped-query decode on the tensor cores (q_per_kv = g >= 2): a CTA serves
// QG <= 16 query heads of one K/V head. The QG queries are the rows of the A
// operand of mma.sync m16n8k16 (rows QG..15 are zero), so every K/V row streamed
// from HBM feeds all QG queries through the MMA instead of QG dot products and
// shuffle reductions on the CUDA cores.
//
// Each of the four warps streams its own blocks of 16 keys (block j of the split
// goes to warp j mod 4) through a three-slot cp.async ring: a lane copies 16-byte
// chunks of K and V rows (ring, window or the new row, chosen per row) and
// stores chunk c of row r at chunk c ^ (r mod 8), so the eight rows an ldmatrix
// phase reads sit in eight different bank groups. Rows past the split's last key
// are zero-filled by the copy (source size 0), which keeps 0 x NaN out of P V.
// Per block: S = Q K^T (K through ldmatrix), online softmax on the S fragments,
// O += P V (P reused from the S registers as the A operand, V through
// ldmatrix.trans). The warps' partials are merged per query head and written to
// the same workspace, for the same combine kernel, as the CUDA-core kernel's.
// ---------------------------------------------------------------------------
constexpr int kMmaBlockKeys = 16;            // keys per warp block (the MMA's N = 2 x 8)
constexpr int kMmaSlots = 3;                 // cp.async slots per warp

template <int D>
constexpr int mma_slot_bytes() { return 2 * kMmaBlockKeys * D * 2; }    // K and V rows of one block
template <int D, int QG>
constexpr int decode_mma_smem_bytes() {
    constexpr int stages = (kDecodeThreads / 32) * kMmaSlots * mma_slot_bytes<D>();
    constexpr int merge = QG * (kDecodeThreads / 32) * (2 + D) * 4;     // reuses the stage bytes
    return stages > merge ? stages : merge;
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void mma_16816(float* c, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                          uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
// 16-byte global -> shared copy; src_bytes = 0 stores zeros and reads nothing
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// byte offset of 16-byte chunk `chunk` of row `row` in a swizzled block
template <int D>
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
    return (uint32_t)(row * (D * 2) + ((chunk ^ (row & 7)) << 4));
}

template <int D, int QG>
__global__ void __launch_bounds__(kDecodeThreads) decode_split_mma_kernel(
        const uint8_t* __restrict__ ring_k, const uint8_t* __restrict__ ring_v, uint4* __restrict__ win_k,
        uint4* __restrict__ win_v, const int32_t* __restrict__ ring_len, const int32_t* __restrict__ win_fill,
        const int32_t* __restrict__ win_idx, const int32_t* __restrict__ ks, int32_t n_windows, int32_t W,
        int32_t H, int32_t C_ring, int32_t C_win, const uint32_t* __restrict__ q, const uint4* __restrict__ k_new,
        const uint4* __restrict__ v_new, float scale_log2, float2* __restrict__ ws_ml, float* __restrict__ ws_o,
        int32_t n_splits, int32_t* status, const int32_t* __restrict__ W_per_window, int32_t q_per_kv) {
    using namespace sm100;
    static_assert(QG >= 2 && QG <= 16, "one query per A row");
    constexpr bool HI = QG > 8;                                      // rows 8..15 hold queries too
    constexpr int CPR = D / 8, ROWB = D * 2, NW = kDecodeThreads / 32, BK = kMmaBlockKeys;
    constexpr int SLOT = mma_slot_bytes<D>(), HALF = SLOT / 2;       // K rows, then V rows
    constexpr int PER_LANE = BK * CPR / 32;                          // chunks per lane per tensor
    const int slices = q_per_kv / QG;
    const int b = blockIdx.z, h = blockIdx.y / slices, slice = blockIdx.y % slices, split = blockIdx.x;
    const int64_t bh = (int64_t)b * H + h;
    const int64_t bhq0 = bh * q_per_kv + (int64_t)slice * QG;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    const int32_t R = ring_len[b], fill = win_fill[b], widx = win_idx[b];
    int32_t Tw = 0;
    const bool state_ok = decode_state_ok(R, fill, widx, ks, n_windows, W, C_ring, C_win, &Tw, W_per_window);
    const int64_t total = (int64_t)R + fill + 1;
    const int64_t s0 = (int64_t)split * kDecodeChunk;
    const int64_t s1 = min(total, s0 + kDecodeChunk);
    if (!state_ok || s0 >= s1) {
        if (!state_ok && split == 0 && blockIdx.y == 0 && tid == 0) report(status, FOCUS_ERR_CAPACITY);
        for (int j = 0; j < QG; ++j) {
            float* wo = ws_o + ((bhq0 + j) * n_splits + split) * D;
            for (int c = tid; c < D; c += blockDim.x) wo[c] = 0.f;
            if (tid == 0) ws_ml[(bhq0 + j) * n_splits + split] = make_float2(-INFINITY, 0.f);
        }
        return;
    }
    if (split == 0 && slice == 0 && tid < CPR) {      // append the new row to the window buffer
        win_k[(bh * C_win + fill) * CPR + tid] = k_new[bh * CPR + tid];
        win_v[(bh * C_win + fill) * CPR + tid] = v_new[bh * CPR + tid];
    }

    extern __shared__ __align__(128) unsigned char smem[];
    const uint32_t my_slots = smem_addr(smem) + (uint32_t)(warp * kMmaSlots * SLOT);
    const uint8_t* rk = ring_k + bh * (int64_t)C_ring * ROWB;
    const uint8_t* rv = ring_v + bh * (int64_t)C_ring * ROWB;
    const uint8_t* wk = reinterpret_cast<const uint8_t*>(win_k) + bh * (int64_t)C_win * ROWB;
    const uint8_t* wv = reinterpret_cast<const uint8_t*>(win_v) + bh * (int64_t)C_win * ROWB;
    const uint8_t* nk = reinterpret_cast<const uint8_t*>(k_new) + bh * ROWB;
    const uint8_t* nv = reinterpret_cast<const uint8_t*>(v_new) + bh * ROWB;

    const int nb = (int)((s1 - s0 + BK - 1) / BK);                    // key blocks in the split
    const int my_nb = nb > warp ? (nb - warp + NW - 1) / NW : 0;      // this warp's: warp, warp + NW, ...
    auto load_block = [&](int i) {                                    // the warp's i-th block into slot i % 3
        const int64_t kb = s0 + (int64_t)(warp + i * NW) * BK;
        const uint32_t dst = my_slots + (uint32_t)((i % kMmaSlots) * SLOT);
#pragma unroll
        for (int u = 0; u < PER_LANE; ++u) {
            const int idx = u * 32 + lane, r = idx / CPR, ch = idx % CPR;
            const int64_t key = kb + r;
            const uint8_t *sk = nk, *sv = nv;                         // the new row (or a zero-filled one)
            if (key < R) {
                sk = rk + key * ROWB;
                sv = rv + key * ROWB;
            } else if (key < (int64_t)R + fill) {
                sk = wk + (key - R) * ROWB;
                sv = wv + (key - R) * ROWB;
            }
            const uint32_t n = key < s1 ? 16u : 0u;
            cp_async16(dst + swz<D>(r, ch), sk + ch * 16, n);
            cp_async16(dst + HALF + swz<D>(r, ch), sv + ch * 16, n);
        }
    };
#pragma unroll
    for (int i = 0; i < kMmaSlots - 1; ++i) {
        if (i < my_nb) load_block(i);
        cp_async_commit();
    }

    const int g = lane >> 2, t4 = lane & 3;                 // fragment rows g, g + 8 and column pair
    // Q as A fragments: rows below QG hold the CTA's query heads, the rest are zero
    uint32_t qa[D / 16][4];
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            const int row = g + 8 * hr;
            const bool live = row < QG;
            const int64_t qw = (bhq0 + (live ? row : 0)) * (D / 2) + kk * 8 + t4;   // 32-bit words of q
            qa[kk][hr] = live ? q[qw] : 0u;
            qa[kk][2 + hr] = live ? q[qw + 4] : 0u;
        }
    }
    float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};   // rows g and g + 8
    float oacc[D / 8][4];
#pragma unroll
    for (int i = 0; i < D / 8; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
    const int mi = lane >> 3;

    for (int i = 0; i < my_nb; ++i) {
        if (i + kMmaSlots - 1 < my_nb) load_block(i + kMmaSlots - 1);   // into the slot read at i - 1
        cp_async_commit();
        cp_async_wait<kMmaSlots - 1>();                                  // block i has landed
        __syncwarp();
        const uint32_t cK = my_slots + (uint32_t)((i % kMmaSlots) * SLOT), cV = cK + HALF;
        const int nrow = (int)min((int64_t)BK, s1 - (s0 + (int64_t)(warp + i * NW) * BK));
        float sacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
            const int key = (mi >> 1) * 8 + (lane & 7);
            uint32_t r0, r1, r2, r3;
            ldsm_x4(cK + swz<D>(key, kk * 2 + (mi & 1)), r0, r1, r2, r3);
            mma_16816(sacc[0], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], r0, r1);
            mma_16816(sacc[1], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], r2, r3);
        }
        // online softmax on rows g (accumulators 0, 1) and g + 8 (2, 3), columns
        // 2 t4 and 2 t4 + 1 of each 8-key half
        uint32_t pa[4] = {0u, 0u, 0u, 0u};                   // P as the A operand of P V
#pragma unroll
        for (int hr = 0; hr < (HI ? 2 : 1); ++hr) {
            float sv[4];
#pragma unroll
            for (int n = 0; n < 2; ++n)
#pragma unroll
                for (int e = 0; e < 2; ++e)
                    sv[n * 2 + e] = n * 8 + 2 * t4 + e < nrow ? sacc[n][2 * hr + e] * scale_log2 : -INFINITY;
            float mx = fmaxf(fmaxf(sv[0], sv[1]), fmaxf(sv[2], sv[3]));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float mn = fmaxf(m[hr], mx);
            const float corr = ex2_approx(m[hr] - mn);       // 0 when m was -inf
            l[hr] *= corr;
#pragma unroll
            for (int d8 = 0; d8 < D / 8; ++d8) { oacc[d8][2 * hr] *= corr; oacc[d8][2 * hr + 1] *= corr; }
            m[hr] = mn;
            float p[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                p[e] = ex2_approx(sv[e] - mn);
                l[hr] += p[e];
            }
            pa[hr] = pack_bf16x2(p[0], p[1]);
            pa[2 + hr] = pack_bf16x2(p[2], p[3]);
        }
#pragma unroll
        for (int dp = 0; dp < D / 16; ++dp) {
            const int key = (mi & 1) * 8 + (lane & 7);
            uint32_t r0, r1, r2, r3;
            ldsm_x4_t(cV + swz<D>(key, 2 * dp + (mi >> 1)), r0, r1, r2, r3);
            mma_16816(oacc[2 * dp], pa[0], pa[1], pa[2], pa[3], r0, r1);
            mma_16816(oacc[2 * dp + 1], pa[0], pa[1], pa[2], pa[3], r2, r3);
        }
        __syncwarp();                                        // slot i % 3 is refilled at i + 1
    }
    cp_async_wait<0>();

    // ---- merge the four warps' partials per query head (in the stage bytes) --
    __syncthreads();
    float* sm_m = reinterpret_cast<float*>(smem);          // [NW][QG]
    float* sm_l = sm_m + NW * QG;                           // [NW][QG]
    float* sm_o = sm_l + NW * QG;                           // [NW][QG][D]
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
        const int row = g + 8 * hr;
        float lr = l[hr];
        lr += __shfl_xor_sync(0xffffffffu, lr, 1);
        lr += __shfl_xor_sync(0xffffffffu, lr, 2);
        if (row < QG) {
            if (t4 == 0) { sm_m[warp * QG + row] = m[hr]; sm_l[warp * QG + row] = lr; }
#pragma unroll
            for (int d8 = 0; d8 < D / 8; ++d8) {
                sm_o[(warp * QG + row) * D + d8 * 8 + 2 * t4] = oacc[d8][2 * hr];
                sm_o[(warp * QG + row) * D + d8 * 8 + 2 * t4 + 1] = oacc[d8][2 * hr + 1];
            }
        }
    }
    __syncthreads();
    for (int col = tid; col < QG * D; col += kDecodeThreads) {
        const int j = col / D, cc = col % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < NW; ++w) M = fmaxf(M, sm_m[w * QG + j]);
        float L = 0.f, A = 0.f;
        if (M != -INFINITY) {
#pragma unroll
            for (int w = 0; w < NW; ++w) {
                const float f = ex2_approx(sm_m[w * QG + j] - M);
                L = fmaf(sm_l[w * QG + j], f, L);
                A = fmaf(sm_o[(w * QG + j) * D + cc], f, A);
            }
        }
        ws_o[((bhq0 + j) * n_splits + split) * D + cc] = A;
        if (cc == 0) ws_ml[(bhq0 + j) * n_splits + split] = make_float2(M, L);
    }
}

template <int D>
__global__ void __launch_bounds__(D) decode_combine_kernel(
        const float2* __restrict__ ws_ml, const float* __restrict__ ws_o, int32_t n_splits, int32_t H,
        __nv_bfloat16* __restrict__ o, float* __restrict__ lse, int32_t* __restrict__ win_fill,
        const int32_t* __restrict__ ring_len, const int32_t* __restrict__ win_idx, const int32_t* __restrict__ ks,
        int32_t n_windows, int32_t W, int32_t C_ring, int32_t C_win, const int32_t* __restrict__ W_per_window) {
    const int b = blockIdx.y, h = blockIdx.x, c = threadIdx.x;   // h: query head, H: query heads
    const int64_t bh = (int64_t)b * H + h;
    const float2* ml = ws_ml + bh * n_splits;
    const float* wo = ws_o + bh * n_splits * D;
    float M = -INFINITY;
    for (int s = 0; s < n_splits; ++s) M = fmaxf(M, ml[s].x);
    float L = 0.f, A = 0.f;
    if (M != -INFINITY) {
        for (int s = 0; s < n_splits; ++s) {
            const float2 x = ml[s];
            if (x.x == -INFINITY) continue;
            const float f = exp2f(x.x - M);
            L = fmaf(x.y, f, L);
            A = fmaf(wo[(int64_t)s * D + c], f, A);
        }
    }
    o[bh * D + c] = __float2bfloat16_rn(L > 0.f ? A / L : 0.f);
    if (c == 0 && lse) lse[bh] = L > 0.f ? (M + log2f(L)) * 0.69314718055994531f : -INFINITY;
    if (h == 0 && c == 0) {
        int32_t Tw = 0;
        if (decode_state_ok(ring_len[b], win_fill[b], win_idx[b], ks, n_windows, W, C_ring, C_win, &Tw,
                            W_per_window))
            win_fill[b] += 1;
    }
}

// Rotary embedding of the new row: q and k_new turn by p theta_i with
// p = pos_base[b] + win_fill[b], the new row's position id. One block per
// (head, sequence), one thread per pair; the rotated rows go to the workspace and
// the split kernel reads them in place of q and k_new.
template <int D>
__global__ void __launch_bounds__(D / 2) decode_rope_kernel(
        const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ k_new,
        __nv_bfloat16* __restrict__ q_rot, __nv_bfloat16* __restrict__ k_rot, const int32_t* __restrict__ pos_base,
        const int32_t* __restrict__ win_fill, int32_t H, int32_t q_per_kv, const __grid_constant__ RopeTable rope) {
    const int b = blockIdx.y, hq = blockIdx.x, i = threadIdx.x;    // grid: query heads x sequences
    const int64_t qrow = ((int64_t)b * H * q_per_kv + hq) * D;
    const int64_t p = (int64_t)pos_base[b] + win_fill[b];
    const float2 cs = rope_cs((double)p * rope.theta[i]);
    const float ql = __bfloat162float(q[qrow + i]), qh = __bfloat162float(q[qrow + i + D / 2]);
    q_rot[qrow + i] = __float2bfloat16_rn(ql * cs.x - qh * cs.y);
    q_rot[qrow + i + D / 2] = __float2bfloat16_rn(qh * cs.x + ql * cs.y);
    if (hq % q_per_kv == 0) {                                      // the K/V head's new key, once
        const int64_t krow = ((int64_t)b * H + hq / q_per_kv) * D;
        const float kl = __bfloat162float(k_new[krow + i]), kh = __bfloat162float(k_new[krow + i + D / 2]);
        k_rot[krow + i] = __float2bfloat16_rn(kl * cs.x - kh * cs.y);
        k_rot[krow + i + D / 2] = __float2bfloat16_rn(kh * cs.x + kl * cs.y);
    }
}

// Workspace: split partials (m, l) and o, then, with the rotary embedding, the
// rotated q and k_new (16-byte aligned).
int32_t q_heads_per_kv(const focus_cache& c) { return c.q_per_kv > 1 ? c.q_per_kv : 1; }

size_t partials_bytes(const focus_cache& c) {
    return (size_t)((int64_t)c.B * c.H * q_heads_per_kv(c) * decode_num_splits(c) * (2 + c.d)) * sizeof(float);
}
size_t rope_rows_offset(const focus_cache& c) { return (partials_bytes(c) + 255) & ~(size_t)255; }

template <int D, int QG>
cudaError_t launch_decode_split(const focus_cache& c, int32_t ns, const void* q, const void* k_new,
                                const void* v_new, float scale, float2* ws_ml, float* ws_o, int32_t* status,
                                cudaStream_t stream) {
    const int32_t g = q_heads_per_kv(c);
    constexpr int smem = decode_smem_bytes<D, QG>();
    cudaError_t e0 = cudaFuncSetAttribute(decode_split_kernel<D, QG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          smem);
    if (e0 != cudaSuccess) return e0;
    decode_split_kernel<D, QG><<<dim3(ns, c.H * (g / QG), c.B), kDecodeThreads + 32, smem, stream>>>(
        (const uint4*)c.ring_k, (const uint4*)c.ring_v, (uint4*)c.win_k, (uint4*)c.win_v, c.ring_len,
        c.win_fill, c.win_idx, c.k_per_window, c.n_windows, c.W, c.H, c.C_ring, c.C_win, (const uint4*)q,
        (const uint4*)k_new, (const uint4*)v_new, scale * 1.4426950408889634f, ws_ml, ws_o, ns, status,
        c.W_per_window, g);
    return cudaGetLastError();
}

template <int D, int QG>
cudaError_t launch_decode_split_mma(const focus_cache& c, int32_t ns, const void* q, const void* k_new,
                                    const void* v_new, float scale, float2* ws_ml, float* ws_o, int32_t* status,
                                    cudaStream_t stream) {
    const int32_t g = q_heads_per_kv(c);
    constexpr int smem = decode_mma_smem_bytes<D, QG>();
    cudaError_t e0 = cudaFuncSetAttribute(decode_split_mma_kernel<D, QG>,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e0 != cudaSuccess) return e0;
    decode_split_mma_kernel<D, QG><<<dim3(ns, c.H * (g / QG), c.B), kDecodeThreads, smem, stream>>>(
        (const uint8_t*)c.ring_k, (const uint8_t*)c.ring_v, (uint4*)c.win_k, (uint4*)c.win_v, c.ring_len,
        c.win_fill, c.win_idx, c.k_per_window, c.n_windows, c.W, c.H, c.C_ring, c.C_win, (const uint32_t*)q,
        (const uint4*)k_new, (const uint4*)v_new, scale * 1.4426950408889634f, ws_ml, ws_o, ns, status,
        c.W_per_window, g);
    return cudaGetLastError();
}

template <int D>
cudaError_t launch_decode_d(const focus_cache& c, const void* q, const void* k_new, const void* v_new,
                            float scale, void* o, float* lse, void* workspace, int32_t* status,
                            cudaStream_t stream) {
    const int32_t ns = decode_num_splits(c);
    const int32_t g = q_heads_per_kv(c);
    const int64_t Hq = (int64_t)c.H * g;
    float2* ws_ml = reinterpret_cast<float2*>(workspace);
    float* ws_o = reinterpret_cast<float*>(ws_ml + (int64_t)c.B * Hq * ns);
    if (c.rope_theta > 0.f) {
        __nv_bfloat16* q_rot = reinterpret_cast<__nv_bfloat16*>((char*)workspace + rope_rows_offset(c));
        __nv_bfloat16* k_rot = q_rot + (int64_t)c.B * Hq * D;
        RopeTable rope;
        rope_table_fill(&rope, D, c.rope_theta);
        decode_rope_kernel<D><<<dim3((unsigned)Hq, c.B), D / 2, 0, stream>>>(
            (const __nv_bfloat16*)q, (const __nv_bfloat16*)k_new, q_rot, k_rot, c.pos_base, c.win_fill, c.H, g,
            rope);
        cudaError_t er = cudaGetLastError();
        if (er != cudaSuccess) return er;
        q = q_rot;
        k_new = k_rot;
    }
    // grouped heads go to the tensor-core kernel (up to sixteen query heads per
    // K/V pass); one query head per K/V head, or an odd group, to the CUDA-core one
    cudaError_t e =
        (g % 16 == 0)  ? launch_decode_split_mma<D, 16>(c, ns, q, k_new, v_new, scale, ws_ml, ws_o, status, stream)
        : (g % 8 == 0) ? launch_decode_split_mma<D, 8>(c, ns, q, k_new, v_new, scale, ws_ml, ws_o, status, stream)
        : (g % 4 == 0) ? launch_decode_split_mma<D, 4>(c, ns, q, k_new, v_new, scale, ws_ml, ws_o, status, stream)
        : (g % 2 == 0) ? launch_decode_split_mma<D, 2>(c, ns, q, k_new, v_new, scale, ws_ml, ws_o, status, stream)
                       : launch_decode_split<D, 1>(c, ns, q, k_new, v_new, scale, ws_ml, ws_o, status, stream);
    if (e != cudaSuccess) return e;
    decode_combine_kernel<D><<<dim3((unsigned)Hq, c.B), D, 0, stream>>>(
        ws_ml, ws_o, ns, (int32_t)Hq, (__nv_bfloat16*)o, lse, c.win_fill, c.ring_len, c.win_idx, c.k_per_window,
        c.n_windows, c.W, c.C_ring, c.C_win, c.W_per_window);
    return cudaGetLastError();
}

}  // namespace

int32_t decode_num_splits(const focus_cache& c) {
    return (int32_t)ceil_div64((int64_t)c.C_ring + c.C_win, kDecodeChunk);
}

size_t decode_workspace_bytes(const focus_cache& c) {
    if (c.rope_theta > 0.f)
        return rope_rows_offset(c) + (size_t)c.B * c.H * (q_heads_per_kv(c) + 1) * c.d * sizeof(__nv_bfloat16);
    return partials_bytes(c);
}

cudaError_t launch_decode(const focus_cache& c, const void* q, const void* k_new, const void* v_new,
                          float scale, void* o, float* lse, void* workspace, int32_t* status,
                          cudaStream_t stream) {
    if (c.d == 128) return launch_decode_d<128>(c, q, k_new, v_new, scale, o, lse, workspace, status, stream);
    return launch_decode_d<64>(c, q, k_new, v_new, scale, o, lse, workspace, status, stream);
}

// Device address of g_decode_scratch on the current device. Host code cannot
// pass the array's name to a kernel (on the host it names a stand-in, not device
// memory), so the first call on each device looks the address up, with that
// device current, and keeps it.
cudaError_t decode_noalloc_scratch(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxScratchDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_decode_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

cudaError_t launch_decode_noalloc(const focus_cache& c, const void* q, const void* k_new, const void* v_new,
                                  float scale, void* o, float* lse, int32_t* status, cudaStream_t stream) {
    void* scratch = nullptr;
    cudaError_t e = decode_noalloc_scratch(&scratch);
    if (e != cudaSuccess) return e;
    return launch_decode(c, q, k_new, v_new, scale, o, lse, scratch, status, stream);
}

}  // namespace focus
