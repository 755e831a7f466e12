// leap_selftest_bounded_wait: the give-up path of the kernels' bounded waits,
// exercised on purpose.  One thread waits, through mbar_wait_bounded (the
// wait every mbarrier of the fused loss and tensor-core kernels uses), on an
// mbarrier that nothing arrives at and no copy completes; with a short limit
// the wait gives up, sets LEAP_DEV_TIMEOUT in the sticky status word and the
// kernel returns.  Nothing is in flight when it does (no copy was issued and
// no tensor memory is held), so the context stays usable.
#include "../../include/leap.h"
#include "leap_common.cuh"
#include "leap_internal.h"

#include <cuda_runtime.h>

namespace leap {
namespace {

__global__ void selftest_wait_kernel(unsigned int* status, uint64_t limit_ns, unsigned long long* waited_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);   // one arrival would complete phase 0; none comes
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const uint64_t t0 = globaltimer_ns();
        const bool done = mbar_wait_bounded<false>(&bar, 0u, status, &abort_flag, limit_ns);
        if (waited_ns) *waited_ns = done ? 0ull : (unsigned long long)(globaltimer_ns() - t0);
    }
}

}  // namespace
}  // namespace leap

extern "C" leap_status_t leap_selftest_bounded_wait(uint64_t limit_ns, uint64_t* waited_ns, void* stream) {
    if (limit_ns < 1000ull || limit_ns > 10000000000ull) return LEAP_ERR_INVALID_ARG;
    unsigned int* status = leap::device_status_ptr();
    if (!status) return LEAP_ERR_CUDA;
    leap::selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
        status, limit_ns, reinterpret_cast<unsigned long long*>(waited_ns));
    return cudaGetLastError() == cudaSuccess ? LEAP_OK : LEAP_ERR_CUDA;
}
