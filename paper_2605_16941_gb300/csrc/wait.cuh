// wait.cuh -- bounded mbarrier waits shared by the kernels that wait on one another's copies or MMAs.
//
// No wait in this library can hang the GPU: each gives up after a time limit
// and raises the CTA's abort flag, so that the CTA's other roles stop waiting
// too.  The kernel then records WINO_ERR_DEVICE_TIMEOUT in the call's status
// word (at a point where that is ordered after the word was cleared), which
// the finish kernel and wino_read_device_status report to the host.
#pragma once

#include <cstdint>

#include "wino.h"
#include "ptx.cuh"

namespace wino {

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s per wait
constexpr uint64_t kDrainLimitNs = 200000000ull;  // 0.2 s for draining after an abort

// Wait for phase `parity` of `bar`; false once `limit_ns` passed (the abort flag is then raised) or another
// role of this CTA aborted.  kCluster: acquire at cluster scope (a barrier the peer CTA of a pair arrives on).
template <bool kCluster = false>
__device__ bool wait_bounded(uint32_t bar, uint32_t parity, int32_t *abort_flag, uint64_t limit_ns = kWaitLimitNs)
{
    auto try_wait = [&] { return kCluster ? ptx::mbar_try_wait_cluster(bar, parity) : ptx::mbar_try_wait(bar, parity); };
    if (try_wait())
        return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        if (try_wait())
            return true;
        if ((it & 15u) == 0) {
            if (*reinterpret_cast<volatile int32_t *>(abort_flag))
                return false;
            if (ptx::globaltimer_ns() - t0 > limit_ns) {
                atomicExch(abort_flag, 1);
                return false;
            }
        }
    }
}

// Bounded wait that ignores the abort flag (used only to drain after an abort).
__device__ inline bool wait_drain(uint32_t bar, uint32_t parity, uint64_t limit_ns = kDrainLimitNs)
{
    const uint64_t t0 = ptx::globaltimer_ns();
    while (!ptx::mbar_try_wait(bar, parity))
        if (ptx::globaltimer_ns() - t0 > limit_ns)
            return false;
    return true;
}

}  // namespace wino
