// acrl_selftest_wait_timeout: exercises the bounded mbarrier wait that guards
// every pipeline wait of the tensor-core kernel, on a barrier that nothing
// ever arrives on.  The wait gives up after the requested time, raises
// ACRL_FLAG_TIMEOUT and the kernel returns: the context stays usable.
#include "acrl_device.cuh"
#include "acrl_host.h"
#include "mbarrier.cuh"

namespace acrl {
namespace {

__global__ void wait_timeout_kernel(int32_t* flags, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    // phase 0 never completes: nobody arrives
    const bool ok = wait_phase(&bar, 0, nullptr, limit_ns);
    if (!ok && threadIdx.x == 0) raise_flag(flags, ACRL_FLAG_TIMEOUT);
}

}  // namespace
}  // namespace acrl

using namespace acrl;

extern "C" acrl_status acrl_selftest_wait_timeout(int32_t* dev_flags, int64_t limit_ns, acrl_stream stream) {
    if (!dev_flags || limit_ns < 0 || limit_ns > int64_t(kWaitNs)) return ACRL_ERR_INVALID_ARG;
    wait_timeout_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(dev_flags, uint64_t(limit_ns));
    return launch_status();
}
