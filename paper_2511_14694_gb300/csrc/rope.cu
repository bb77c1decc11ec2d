// Rotary position embedding of a prefill span's q and k rows, as a pass of its
// own ahead of the attention (RoFormer rotation with rotate-half pairing at the
// layout's position ids: Sec. 3.2 gives every row, FOCUS rows included, a real
// position, and row i of the span sits at position win_off[w_begin] + i).
//
// The rotation is elementwise and bound by HBM (q and k read once, their rotated
// copies written once); the attention that follows is bound by the tensor cores.
// As separate launches each runs at its own roofline; done inside the attention
// kernel, the rotation had two warps per SM and the registers left over from the
// attention, and it held the attention's producer back.
//
// Thread (row i, chunk j) owns the pairs 8j .. 8j + 7 of row i: the 16-byte chunk j
// of the row's first half and its partner chunk D/2 columns on. Their angles
// p theta_e are formed once per thread (fp64 product reduced modulo 2 pi, then
// fp32 sin/cos: positions reach ~10^6, where an fp32 product would be off by
// ~0.1 rad) and turn that chunk pair in every (sequence, head) of q and of k.
// A warp covers four whole rows (1 KB contiguous) per (sequence, head).
#include "prefill_tc_common.cuh"

namespace focus {
namespace prefill {
namespace {

constexpr int kRopeThreads = 256;
constexpr int kRopeUnroll = 4;                       // (sequence, head) rows in flight per thread

template <int D>
__global__ void __launch_bounds__(kRopeThreads) rope_rotate_kernel(
        const __grid_constant__ RopeTable t, const uint4* __restrict__ q_src, const uint4* __restrict__ k_src,
        uint4* __restrict__ q_dst, uint4* __restrict__ k_dst, int64_t T_span, int32_t BHq, int32_t BHk,
        const int32_t* __restrict__ win_off, int32_t w_begin) {
    constexpr int HALF = D / 16;                       // 16-byte chunks in half a row
    constexpr int CPR = D / 8;                         // 16-byte chunks in a row
    constexpr int ROWS = kRopeThreads / HALF;          // rows per block
    const int j = threadIdx.x % HALF;
    const int64_t row = (int64_t)blockIdx.x * ROWS + threadIdx.x / HALF;
    if (row >= T_span) return;
    const double p = (double)((int64_t)win_off[w_begin] + row);
    float2 cs[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) cs[e] = rope_cs(p * t.theta[8 * j + e]);
    const Rot8 r = rot8_make(cs);
    const int64_t stride = T_span * CPR;               // chunks per (sequence, head)
    const int64_t at = row * CPR + j;
#pragma unroll 1
    for (int set = 0; set < 2; ++set) {
        const uint4* src = (set == 0 ? q_src : k_src) + at;
        uint4* dst = (set == 0 ? q_dst : k_dst) + at;
        const int32_t n = set == 0 ? BHq : BHk;
        int32_t h = 0;
#pragma unroll 1
        for (; h + kRopeUnroll <= n; h += kRopeUnroll) {
            uint4 lo[kRopeUnroll], hi[kRopeUnroll];
#pragma unroll
            for (int u = 0; u < kRopeUnroll; ++u) {
                lo[u] = __ldcs(src + (int64_t)(h + u) * stride);
                hi[u] = __ldcs(src + (int64_t)(h + u) * stride + HALF);
            }
#pragma unroll
            for (int u = 0; u < kRopeUnroll; ++u) {
                rot8_apply(lo[u], hi[u], r);
                dst[(int64_t)(h + u) * stride] = lo[u];
                dst[(int64_t)(h + u) * stride + HALF] = hi[u];
            }
        }
#pragma unroll 1
        for (; h < n; ++h) {
            uint4 lo = __ldcs(src + (int64_t)h * stride), hi = __ldcs(src + (int64_t)h * stride + HALF);
            rot8_apply(lo, hi, r);
            dst[(int64_t)h * stride] = lo;
            dst[(int64_t)h * stride + HALF] = hi;
        }
    }
}

template <int D>
cudaError_t launch_d(const focus_cache& c, const focus_prefill_args& a, void* q_rot, void* k_rot,
                     cudaStream_t stream) {
    constexpr int ROWS = kRopeThreads / (D / 16);
    const int32_t g = c.q_per_kv > 1 ? c.q_per_kv : 1;
    RopeTable t;
    rope_table_fill(&t, D, c.rope_theta);
    const int64_t blocks = (a.T_span + ROWS - 1) / ROWS;
    rope_rotate_kernel<D><<<(unsigned)blocks, kRopeThreads, 0, stream>>>(
        t, (const uint4*)a.q, (const uint4*)a.k, (uint4*)q_rot, (uint4*)k_rot, a.T_span, c.B * c.H * g, c.B * c.H,
        a.d_win_off, a.w_begin);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rope_rotate(const focus_cache& c, const focus_prefill_args& a, void* q_rot, void* k_rot,
                               cudaStream_t stream) {
    if (a.T_span <= 0) return cudaSuccess;
    return c.d == 128 ? launch_d<128>(c, a, q_rot, k_rot, stream) : launch_d<64>(c, a, q_rot, k_rot, stream);
}

}  // namespace prefill
}  // namespace focus
