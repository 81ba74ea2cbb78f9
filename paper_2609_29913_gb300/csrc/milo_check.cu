// milo_check.cu -- a check of the bounded wait that every kernel of the
// library uses: one warp waits on an mbarrier that nothing completes (or that
// it completes itself first) through mbar_wait, with a short limit.  A wait
// that runs out sets MILO_ERR_TIMEOUT in the status word and returns, and the
// kernel ends normally, so a failed wait is reported without faulting or
// hanging the GPU; the host reads the word with milo_get_device_status.
#include "milo.h"
#include "milo_internal.h"
#include "milo_ptx.cuh"

namespace milo {
namespace {

__global__ void __launch_bounds__(32) wait_check_kernel(int32_t *status, uint64_t limit_ns, int arrive)
{
    __shared__ __align__(8) uint64_t bar;
    const uint32_t b = smem_u32(&bar);
    if (threadIdx.x == 0) {
        mbar_init(b, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    if (arrive && threadIdx.x == 0) mbar_arrive(b);
    __syncwarp();
    mbar_wait(b, 0, status, limit_ns);
}

}  // namespace

cudaError_t launch_wait_check(int32_t *status, uint64_t limit_ns, int arrive, cudaStream_t stream)
{
    wait_check_kernel<<<1, 32, 0, stream>>>(status, limit_ns, arrive);
    return cudaGetLastError();
}

}  // namespace milo
