// Windowed prefill attention over the compressed context, legacy tensor-core
// path (mma.sync m16n8k16 bf16, fp32 accumulate). Kept as the comparison
// baseline for the tcgen05/TMEM kernel.
//
// Row a of window w attends to ring[0, ring_off[w]) (retained FOCUS K/V of all
// earlier windows, fully visible) and to window rows [0, a] (causal): Eq.
// focus-attn's visible set, App. A.1-A.2. The mask is analytic per key tile:
// only the last partial ring tile (keys >= R_w) and the diagonal window tile
// (key > row) are masked; no mask tensor exists.
//
// CTA = 4 warps x 16 query rows (BM = 64), key tiles of BN = 64 rows,
// cp.async double buffering, XOR-swizzled shared memory for ldmatrix,
// FlashAttention-2-style online softmax in registers (log2 domain).
#include "common.cuh"

namespace focus {
namespace {

constexpr int BM = 64, BN = 64, kThreads = 128;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
    const int n = valid ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// Swizzled element offset of (row, 16-byte chunk) in a [rows][D] bf16 tile.
template <int D>
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
    return (uint32_t)(row * D + ((chunk ^ (row & 7)) << 3));
}

template <int D>
__device__ __forceinline__ void load_tile(__nv_bfloat16* s, const __nv_bfloat16* base, int valid_rows) {
    constexpr int CH = D / 8;
    for (int i = threadIdx.x; i < BN * CH; i += kThreads) {
        const int r = i / CH, c = i % CH;
        const bool v = r < valid_rows;
        const __nv_bfloat16* src = v ? base + (int64_t)r * D + c * 8 : base;
        cp_async16(smem_u32(s + swz<D>(r, c)), src, v);
    }
}

template <int D>
__global__ void __launch_bounds__(kThreads) prefill_mma_kernel(
        const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ k,
        const __nv_bfloat16* __restrict__ v, const __nv_bfloat16* __restrict__ ring_k,
        const __nv_bfloat16* __restrict__ ring_v, __nv_bfloat16* __restrict__ o, float* __restrict__ lse,
        int64_t T_span, const int32_t* __restrict__ win_off, const int32_t* __restrict__ ring_off,
        int32_t w_begin, int32_t w_end, int32_t tiles_pw, int32_t H, int32_t C_ring, float scale_log2,
        int32_t* status) {
    constexpr int CH = D / 8;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem_raw);
    __nv_bfloat16* sK = sQ + BM * D;        // [2][BN][D]
    __nv_bfloat16* sV = sK + 2 * BN * D;    // [2][BN][D]

    // Longest work first: later windows carry longer rings; later tiles more keys.
    const int32_t wi = blockIdx.x / tiles_pw;
    const int32_t tile = tiles_pw - 1 - (int32_t)(blockIdx.x % tiles_pw);
    const int32_t w = w_end - 1 - wi;
    const int h = blockIdx.y, b = blockIdx.z;
    const int64_t bh = (int64_t)b * H + h;
    const int32_t w0 = win_off[w_begin];
    const int32_t Tw = win_off[w + 1] - win_off[w];
    const int32_t a0 = tile * BM;
    if (a0 >= Tw) return;
    const int32_t Rw = ring_off[w];
    if (Rw > C_ring || (int64_t)(win_off[w_end] - w0) > T_span) {
        if (threadIdx.x == 0) report(status, FOCUS_ERR_CAPACITY);
        return;
    }
    const int64_t row_base = (int64_t)(win_off[w] - w0);   // window's first row in the span tensors
    const __nv_bfloat16* qh = q + (bh * T_span + row_base) * D;
    const __nv_bfloat16* kh = k + (bh * T_span + row_base) * D;
    const __nv_bfloat16* vh = v + (bh * T_span + row_base) * D;
    const __nv_bfloat16* rkh = ring_k + bh * (int64_t)C_ring * D;
    const __nv_bfloat16* rvh = ring_v + bh * (int64_t)C_ring * D;

    const int n_ring = (Rw + BN - 1) / BN;
    const int n_tiles = n_ring + tile + 1;

    auto issue = [&](int it, int buf) {
        const __nv_bfloat16 *kb, *vb;
        int valid;
        if (it < n_ring) {
            kb = rkh + (int64_t)it * BN * D;
            vb = rvh + (int64_t)it * BN * D;
            valid = min(BN, Rw - it * BN);
        } else {
            const int t = it - n_ring;
            kb = kh + (int64_t)t * BN * D;
            vb = vh + (int64_t)t * BN * D;
            valid = min(BN, Tw - t * BN);
        }
        load_tile<D>(sK + buf * BN * D, kb, valid);
        load_tile<D>(sV + buf * BN * D, vb, valid);
    };

    // Q tile + first K/V tile
    {
        const int valid = min(BM, Tw - a0);
        for (int i = threadIdx.x; i < BM * CH; i += kThreads) {
            const int r = i / CH, c = i % CH;
            const bool ok = r < valid;
            const __nv_bfloat16* src = ok ? qh + (int64_t)(a0 + r) * D + c * 8 : qh;
            cp_async16(smem_u32(sQ + swz<D>(r, c)), src, ok);
        }
        issue(0, 0);
        cp_async_commit();
    }

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane >> 2, t4 = lane & 3;

    uint32_t qf[D / 16][4];
    float oacc[D / 8][4];
#pragma unroll
    for (int i = 0; i < D / 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) oacc[i][j] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

    const int qrow0 = a0 + warp * 16 + g;        // in-window row of c0/c1
    const int qrow1 = qrow0 + 8;                  // in-window row of c2/c3

    for (int it = 0; it < n_tiles; ++it) {
        const int buf = it & 1;
        if (it + 1 < n_tiles) {
            issue(it + 1, buf ^ 1);
            cp_async_commit();
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
        __syncthreads();
        if (it == 0) {
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
                const int row = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                const int ch = kk * 2 + (lane >> 4);
                ldsm_x4(smem_u32(sQ + swz<D>(row, ch)), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
            }
        }
        const __nv_bfloat16* cK = sK + buf * BN * D;
        const __nv_bfloat16* cV = sV + buf * BN * D;

        float s[BN / 8][4];
#pragma unroll
        for (int n = 0; n < BN / 8; ++n)
#pragma unroll
            for (int j = 0; j < 4; ++j) s[n][j] = 0.f;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
            for (int np = 0; np < BN / 16; ++np) {
                const int mi = lane >> 3;
                const int key = (2 * np + (mi >> 1)) * 8 + (lane & 7);
                const int ch = kk * 2 + (mi & 1);
                uint32_t r0, r1, r2, r3;
                ldsm_x4(smem_u32(cK + swz<D>(key, ch)), r0, r1, r2, r3);
                mma_bf16(s[2 * np], qf[kk], r0, r1);
                mma_bf16(s[2 * np + 1], qf[kk], r2, r3);
            }
        }

        // analytic mask
        const bool ring_tile = it < n_ring;
        const int kbase = ring_tile ? it * BN : (it - n_ring) * BN;
        const bool need_mask = ring_tile ? (kbase + BN > Rw) : (it - n_ring == tile);
#pragma unroll
        for (int n = 0; n < BN / 8; ++n) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float x = s[n][j] * scale_log2;
                if (need_mask) {
                    const int key = kbase + n * 8 + 2 * t4 + (j & 1);
                    const int row = (j < 2) ? qrow0 : qrow1;
                    const bool vis = ring_tile ? (key < Rw) : (key <= row);
                    if (!vis) x = -INFINITY;
                }
                s[n][j] = x;
            }
        }
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int n = 0; n < BN / 8; ++n) {
            mx0 = fmaxf(mx0, fmaxf(s[n][0], s[n][1]));
            mx1 = fmaxf(mx1, fmaxf(s[n][2], s[n][3]));
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        const float mu0 = mn0 == -INFINITY ? 0.f : mn0, mu1 = mn1 == -INFINITY ? 0.f : mn1;
        const float c0 = exp2f(m0 - mu0), c1 = exp2f(m1 - mu1);
        m0 = mn0;
        m1 = mn1;
        l0 *= c0;
        l1 *= c1;
#pragma unroll
        for (int i = 0; i < D / 8; ++i) {
            oacc[i][0] *= c0; oacc[i][1] *= c0;
            oacc[i][2] *= c1; oacc[i][3] *= c1;
        }
        uint32_t pa[BN / 16][4];
#pragma unroll
        for (int n = 0; n < BN / 8; ++n) {
            const float p0 = exp2f(s[n][0] - mu0), p1 = exp2f(s[n][1] - mu0);
            const float p2 = exp2f(s[n][2] - mu1), p3 = exp2f(s[n][3] - mu1);
            l0 += p0 + p1;
            l1 += p2 + p3;
            pa[n >> 1][(n & 1) * 2 + 0] = pack_bf16(p0, p1);
            pa[n >> 1][(n & 1) * 2 + 1] = pack_bf16(p2, p3);
        }
#pragma unroll
        for (int j = 0; j < BN / 16; ++j) {
#pragma unroll
            for (int dp = 0; dp < D / 16; ++dp) {
                const int mi = lane >> 3;
                const int key = 16 * j + (mi & 1) * 8 + (lane & 7);
                const int ch = 2 * dp + (mi >> 1);
                uint32_t r0, r1, r2, r3;
                ldsm_x4_t(smem_u32(cV + swz<D>(key, ch)), r0, r1, r2, r3);
                mma_bf16(oacc[2 * dp], pa[j], r0, r1);
                mma_bf16(oacc[2 * dp + 1], pa[j], r2, r3);
            }
        }
        __syncthreads();
    }

    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    const float il0 = l0 > 0.f ? 1.f / l0 : 0.f, il1 = l1 > 0.f ? 1.f / l1 : 0.f;

    // Stage the warp's 16 output rows in its own slice of sQ, then store 16 B per lane.
#pragma unroll
    for (int i = 0; i < D / 8; ++i) {
        const int col = i * 8 + 2 * t4;
        const int r0 = warp * 16 + g, r1 = r0 + 8;
        *reinterpret_cast<uint32_t*>(sQ + swz<D>(r0, col >> 3) + (col & 7)) = pack_bf16(oacc[i][0] * il0, oacc[i][1] * il0);
        *reinterpret_cast<uint32_t*>(sQ + swz<D>(r1, col >> 3) + (col & 7)) = pack_bf16(oacc[i][2] * il1, oacc[i][3] * il1);
    }
    __syncwarp();
    __nv_bfloat16* oh = o + (bh * T_span + row_base) * D;
    for (int i = lane; i < 16 * CH; i += 32) {
        const int r = i / CH, c = i % CH;
        const int row = warp * 16 + r;
        if (a0 + row < Tw)
            *reinterpret_cast<uint4*>(oh + (int64_t)(a0 + row) * D + c * 8) =
                *reinterpret_cast<const uint4*>(sQ + swz<D>(row, c));
    }
    if (lse && t4 == 0) {
        float* lh = lse + bh * T_span + row_base;
        constexpr float kLn2 = 0.69314718055994531f;
        if (qrow0 < Tw) lh[qrow0] = l0 > 0.f ? (m0 + log2f(l0)) * kLn2 : -INFINITY;
        if (qrow1 < Tw) lh[qrow1] = l1 > 0.f ? (m1 + log2f(l1)) * kLn2 : -INFINITY;
    }
}

template <int D>
cudaError_t launch_d(const focus_cache& c, const focus_prefill_args& a, int32_t* status, cudaStream_t stream) {
    const int tiles_pw = (a.max_rows + BM - 1) / BM;
    const size_t smem = (size_t)(BM + 4 * BN) * D * sizeof(__nv_bfloat16);
    cudaError_t e = cudaFuncSetAttribute(prefill_mma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((a.w_end - a.w_begin) * tiles_pw), c.H, c.B);
    prefill_mma_kernel<D><<<grid, kThreads, smem, stream>>>(
        (const __nv_bfloat16*)a.q, (const __nv_bfloat16*)a.k, (const __nv_bfloat16*)a.v,
        (const __nv_bfloat16*)c.ring_k, (const __nv_bfloat16*)c.ring_v, (__nv_bfloat16*)a.o, a.lse, a.T_span,
        a.d_win_off, a.d_ring_off, a.w_begin, a.w_end, tiles_pw, c.H, c.C_ring,
        a.scale * 1.4426950408889634f, status);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefill_mma(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                               cudaStream_t stream) {
    if (c.d == 128) return launch_d<128>(c, a, status, stream);
    return launch_d<64>(c, a, status, stream);
}

}  // namespace focus
