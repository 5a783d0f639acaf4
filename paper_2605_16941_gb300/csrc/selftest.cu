// selftest.cu -- device self-test of the bounded-wait failure path.
//
// One CTA initialises an mbarrier that nothing will ever arrive on and waits
// for it with the same bounded wait the score kernel uses, shortened to the
// caller's limit.  The wait must give up and raise the abort flag; the kernel
// records WINO_ERR_DEVICE_TIMEOUT in *status and exits normally, so the CUDA
// context stays usable.  This is how the library's timeout handling is
// exercised on a GPU without hanging or faulting it.
#include "internal.h"
#include "ptx.cuh"
#include "wait.cuh"

namespace wino {
namespace {

__global__ void wait_timeout_kernel(int32_t *status, uint64_t limit_ns)
{
    __shared__ __align__(8) uint64_t bar;
    __shared__ int32_t abort_flag;
    if (threadIdx.x != 0)
        return;
    *status = WINO_OK;
    abort_flag = 0;
    const uint32_t b = ptx::smem_u32(&bar);
    ptx::mbar_init(b, 1);
    ptx::fence_barrier_init();
    // nothing arrives: phase 0 never completes
    if (!wait_bounded(b, 0, &abort_flag, limit_ns) && abort_flag)
        *status = WINO_ERR_DEVICE_TIMEOUT;
}

}  // namespace
}  // namespace wino

extern "C" int wino_selftest_wait_timeout(int32_t *status, int64_t limit_ns, void *stream)
{
    if (!status || limit_ns < 1000 || limit_ns > 1000000000)  // 1 us .. 1 s
        return WINO_ERR_ARG;
    wino::wait_timeout_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(status, (uint64_t)limit_ns);
    return cudaGetLastError() == cudaSuccess ? WINO_OK : WINO_ERR_CUDA;
}
