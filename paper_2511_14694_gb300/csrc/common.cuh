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

// Kernel launchers (one translation unit each).
cudaError_t launch_layout(int64_t N, int32_t W, int32_t M, const int32_t* d_k, bool close_tail,
                          int32_t tail, int32_t B, const uint8_t* d_nt, const focus_layout_out& out,
                          int32_t* status, cudaStream_t stream);

cudaError_t launch_compact_bulk(const focus_cache& c, const focus_compact_args& a, int32_t* status,
                                cudaStream_t stream);
cudaError_t launch_compact_window(const focus_cache& c, int32_t* status, cudaStream_t stream);

int32_t decode_num_splits(const focus_cache& c);
cudaError_t launch_decode(const focus_cache& c, const void* q, const void* k_new, const void* v_new,
                          float scale, void* o, float* lse, void* workspace, int32_t* status,
                          cudaStream_t stream);

cudaError_t launch_decode_noalloc(const focus_cache& c, const void* q, const void* k_new, const void* v_new,
                                  float scale, void* o, float* lse, int32_t* status, cudaStream_t stream);

cudaError_t launch_prefill_mma(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                               cudaStream_t stream);
cudaError_t launch_prefill_tc(const focus_cache& c, const focus_prefill_args& a, int32_t* status,
                              cudaStream_t stream);

}  // namespace focus
