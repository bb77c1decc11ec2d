// Input rows of the augmented sequence (Sec. 3.2 "Setup and tokens"; App. A):
// out[i] = table[tok[i]], where tok is the token stream of the layout (nucleotide
// ids 0..3 and the FOCUS summary token) and table holds one embedding row per
// token id, the summary token's among them.
//
// HBM-bound: the table (n_tokens x D bf16, a few KB to a few tens of KB) stays in
// L1/L2; every output byte is written once. One warp per row (rows strided over
// all warps of the grid), lanes over the row's 16-byte chunks, so each warp
// store covers 512 contiguous bytes; the row's token is one broadcast load.
#include "common.cuh"

namespace focus {
namespace {

__global__ void __launch_bounds__(256) embed_tokens_kernel(const uint8_t* __restrict__ tok, int64_t n_rows,
                                                          const uint4* __restrict__ table, int32_t n_tokens,
                                                          int32_t chunks, uint4* __restrict__ out,
                                                          int32_t* status) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t row = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; row < n_rows; row += warps) {
        const int32_t t = tok[row];
        uint4* o = out + row * chunks;
        if (t < n_tokens) {
            const uint4* src = table + (int64_t)t * chunks;
            for (int32_t c = lane; c < chunks; c += 32) __stcs(&o[c], __ldg(&src[c]));
        } else {
            if (lane == 0) report(status, FOCUS_ERR_INVALID_ARG);
            for (int32_t c = lane; c < chunks; c += 32) __stcs(&o[c], make_uint4(0u, 0u, 0u, 0u));
        }
    }
}

}  // namespace

cudaError_t launch_embed_tokens(const uint8_t* tok, int64_t n_rows, const void* table, int32_t n_tokens, int32_t D,
                                void* out, int32_t* status, cudaStream_t stream) {
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const int32_t chunks = D / 8;
    const int64_t want = (n_rows + 7) / 8;           // 8 warps (rows) per block
    const int64_t cap = (int64_t)sms * 8;            // 8 resident blocks of 256 threads per SM
    const unsigned grid = (unsigned)(want < cap ? want : cap);
    embed_tokens_kernel<<<grid, 256, 0, stream>>>(tok, n_rows, (const uint4*)table, n_tokens, chunks, (uint4*)out,
                                                  status);
    return cudaGetLastError();
}

}  // namespace focus
