// Internal helpers shared by the FOCUS CUDA kernels (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "focus.h"

namespace focus {

// Sticky device status: the first error code wins; later ones are dropped.
__device__ __forceinline__ void report(int32_t* status, int32_t code) {
    if (status) atomicCAS(status, (int32_t)FOCUS_OK, code);
}

__host__ __device__ __forceinline__ int64_t ceil_div64(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Augmented rows of a window of n bases with cadence k: n + B_w, where
// B_w = ceil(n/k) if the window's final partial k-mer is closed, floor(n/k)
// otherwise, and 0 when k == 0 (App. A).
__host__ __device__ __forceinline__ int64_t window_rows(int64_t n, int32_t k, bool close_partial) {
    if (k <= 0) return n;
    int64_t b = close_partial ? (n + k - 1) / k : n / k;
    return n + b;
}

// In-window augmented offset of the j-th FOCUS row of a full window of W bases
// with cadence k > 0: a full k-mer j ends at row (j+1)(k+1)-1; the summary of a
// trailing partial k-mer is the window's last row.
__host__ __device__ __forceinline__ int32_t window_summary_row(int32_t j, int32_t W, int32_t k) {
    if ((int64_t)(j + 1) * k <= W) return (j + 1) * (k + 1) - 1;
    return (int32_t)window_rows(W, k, true) - 1;
}

// First base of the boundary tail of an n-base window (bases at or after it are
// kept with the FOCUS rows); tail = 0 means none.
__host__ __device__ __forceinline__ int64_t tail_start(int64_t n, int32_t tail) {
    return tail > 0 ? (n - tail > 0 ? n - tail : 0) : n;
}

// ---------------------------------------------------------------- rotary embedding
// RoFormer rotation with rotate-half pairing at the layout's position ids: the
// pair (x_i, x_{i+d/2}), i < d/2, turns by p * theta_i, theta_i = base^(-2i/d).
// Positions reach ~10^6, where an fp32 angle p * theta_i is off by up to ~0.1 rad,
// so every angle a kernel starts from is formed and reduced modulo 2 pi in fp64
// and only the reduced angle goes to the fp32 sin/cos. Along a tile, rows step by
// small fixed offsets (|angle| <= 16 rad, accurate in fp32), so a kernel needs one
// fp64 angle per pair and tile start, not per element.
constexpr int kRopeMaxPairs = 64;         // d/2 for d <= 128

// The frequencies, computed once on the host in fp64 (a 512-byte kernel argument).
struct RopeTable {
    double theta[kRopeMaxPairs];          // theta_i
};

// Host: fill the table for head dimension d (even, <= 128) and base > 0.
void rope_table_fill(RopeTable* t, int d, float base);

// (cos, sin) of the fp64 angle a, reduced to [-pi, pi] in fp64 first.
__device__ __forceinline__ float2 rope_cs(double a) {
    const double two_pi = 6.283185307179586476925286766559;
    const double r = a - two_pi * rint(a * (1.0 / two_pi));
    float s, c;
    __sincosf((float)r, &s, &c);
    return make_float2(c, s);
}

// (c1 + i s1)(c2 + i s2): the rotation by the sum of two angles.
__device__ __forceinline__ float2 rope_mul(float2 a, float2 b) {
    return make_float2(a.x * b.x - a.y * b.y, a.y * b.x + a.x * b.y);
}

// Rotate eight pairs held as two 16-byte chunks of bf16 (lo: x_i.., hi: x_{i+d/2}..).
__device__ __forceinline__ void rope_rotate8(uint4& lo, uint4& hi, const float2* cs) {
    __nv_bfloat162* l = reinterpret_cast<__nv_bfloat162*>(&lo);
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&hi);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float2 a = __bfloat1622float2(l[e]), b = __bfloat1622float2(h[e]);
        const float2 c0 = cs[2 * e], c1 = cs[2 * e + 1];
        l[e] = __floats2bfloat162_rn(a.x * c0.x - b.x * c0.y, a.y * c1.x - b.y * c1.y);
        h[e] = __floats2bfloat162_rn(b.x * c0.x + a.x * c0.y, b.y * c1.x + a.y * c1.y);
    }
}

// Kernel launchers (one translation unit each).
// d_W: per-window lengths (device) or NULL for windows of W bases.
cudaError_t launch_layout(int64_t N, int32_t W, const int32_t* d_W, int32_t M, const int32_t* d_k, bool close_tail,
                          int32_t tail, int32_t B, const uint8_t* d_nt, const focus_layout_out& out,
                          int32_t* status, cudaStream_t stream);

// Length of window w of a cache: the schedule's entry, or the fixed W.
__device__ __forceinline__ int32_t cache_window_len(const int32_t* W_per_window, int32_t W, int32_t w) {
    return W_per_window ? W_per_window[w] : W;
}

cudaError_t launch_compact_bulk(const focus_cache& c, const focus_compact_args& a, int32_t* status,
                                cudaStream_t stream);
cudaError_t launch_compact_bulk_rope(const focus_cache& c, const focus_compact_args& a, int32_t* status,
                                     cudaStream_t stream);
cudaError_t launch_compact_window(const focus_cache& c, int32_t* status, cudaStream_t stream);
cudaError_t launch_selftest_timeout(uint64_t limit_ns, int32_t* status, cudaStream_t stream);
cudaError_t launch_embed_tokens(const uint8_t* tok, int64_t n_rows, const void* table, int32_t n_tokens, int32_t D,
                                void* out, int32_t* status, cudaStream_t stream);

int32_t decode_num_splits(const focus_cache& c);
size_t decode_workspace_bytes(const focus_cache& c);
cudaError_t launch_decode(const focus_cache& c, const void* q, const void* k_new, const void* v_new,
                          float scale, void* o, float* lse, void* workspace, int32_t* status,
                          cudaStream_t stream);

cudaError_t launch_decode_noalloc(const focus_cache& c, const void* q, const void* k_new, const void* v_new,
                                  float scale, void* o, float* lse, int32_t* status, cudaStream_t stream);

cudaError_t launch_prefill_mma(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                               cudaStream_t stream);
// FOCUS_PREFILL_KERNEL_* that launch_prefill_tc (or the legacy flag) selects.
int32_t prefill_kernel_choice(const focus_cache& c, const focus_prefill_args& a);
// Workspace bytes the fastest prefill kernel wants for these arguments (0: none).
size_t prefill_workspace_bytes(const focus_cache& c, const focus_prefill_args& a);
cudaError_t launch_prefill_tc(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                              cudaStream_t stream);

}  // namespace focus
