// Self-test of the failure path: a bounded mbarrier wait that nothing completes
// gives up and reports FOCUS_ERR_TIMEOUT in the device status word, exactly as a
// kernel whose TMA copies or MMAs never arrive would, and the context stays usable.
// No fault, no unbounded spin: the wait is the library's own mbar_wait.
#include "common.cuh"
#include "sm100.cuh"

namespace focus {
namespace {

__global__ void __launch_bounds__(32) selftest_timeout_kernel(uint64_t limit_ns, int32_t* status) {
    using namespace sm100;
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_addr(&bar), 1);         // one arrival would complete phase 0; none comes
        fence_barrier_init();
    }
    __syncwarp();
    if (threadIdx.x == 0 && !mbar_wait(smem_addr(&bar), 0, limit_ns)) report(status, FOCUS_ERR_TIMEOUT);
}

}  // namespace

cudaError_t launch_selftest_timeout(uint64_t limit_ns, int32_t* status, cudaStream_t stream) {
    selftest_timeout_kernel<<<1, 32, 0, stream>>>(limit_ns, status);
    return cudaGetLastError();
}

}  // namespace focus
