// osd_health.cu -- a check of the failure path the kernels share: the bounded
// mbarrier wait that guards every staging copy (osd_rowspan.cuh).  One thread
// waits on a barrier that nothing completes; when the limit passes it reports
// OSD_ERR_TIMEOUT the way a timed-out staging copy does, and the context stays
// usable.  No logits are read and no copy is in flight.
#include <cstdint>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"

namespace osd {

__global__ void bounded_wait_check_kernel(uint64_t limit_ns, int32_t* status, uint64_t* waited_ns) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);  // expects one arrival, and none comes
    const uint64_t t0 = global_ns();
    const bool done = mbar_wait_bounded(&bar, 0, limit_ns);
    const uint64_t t1 = global_ns();
    *status = done ? static_cast<int32_t>(OSD_OK) : static_cast<int32_t>(OSD_ERR_TIMEOUT);
    if (waited_ns) *waited_ns = t1 - t0;
}

}  // namespace osd

extern "C" osd_status osd_check_bounded_wait(uint32_t limit_us, int32_t* status, uint64_t* waited_ns,
                                             void* stream) {
    using namespace osd;
    if (!status || limit_us == 0 || limit_us > 10000000u) return OSD_ERR_INVALID_ARG;
    if (!aligned_to(status, 4) || (waited_ns && !aligned_to(waited_ns, 8))) return OSD_ERR_INVALID_ARG;
    return from_cuda(launch(bounded_wait_check_kernel, dim3(1), dim3(32), 0, static_cast<cudaStream_t>(stream), 1,
                            static_cast<uint64_t>(limit_us) * 1000ull, status, waited_ns));
}
