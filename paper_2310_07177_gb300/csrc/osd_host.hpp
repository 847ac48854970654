// osd_host.hpp -- host-side helpers shared by the launchers: status mapping,
// argument checks and cluster launches through cudaLaunchKernelEx.
#pragma once

#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdint>

#include "osd.h"

namespace osd {

inline osd_status from_cuda(cudaError_t e) { return e == cudaSuccess ? OSD_OK : OSD_ERR_CUDA; }

inline bool aligned_to(const void* p, size_t a) {
    return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

inline size_t dtype_size(osd_dtype d) { return d == OSD_BF16 ? 2 : 4; }

// exp(x / T) = 2^(x * c) with c = log2(e) / T, carried as c_hi + c_lo where both
// halves are positive floats: the pair removes the rounding of c from every
// exponent argument, and positive halves keep -inf inputs at -inf.
inline void split_scale(float temperature, float* c_hi, float* c_lo) {
    const double c = 1.4426950408889634074 / static_cast<double>(temperature);
    float hi = static_cast<float>(c);
    if (static_cast<double>(hi) > c) hi = std::nextafter(hi, 0.0f);
    float lo = static_cast<float>(c - static_cast<double>(hi));
    if (!(lo > 0.0f)) lo = 1e-30f;
    *c_hi = hi;
    *c_lo = lo;
}

// Streaming multiprocessors of the current device, looked up once per device
// (0 when the query fails).
inline int device_sms() {
    static std::atomic<int> sms[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    int n = sms[dev].load(std::memory_order_relaxed);
    if (n == 0 && cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
        sms[dev].store(n, std::memory_order_relaxed);
    return n;
}

// Launch `kernel` with an optional thread-block cluster of `cluster` CTAs
// along x (cluster == 1 launches without the attribute); launch_ex can also
// mark it a programmatic dependent of the previous kernel on the stream.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_ex(bool dependent, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t stream, int cluster, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    unsigned n = 0;
    if (cluster > 1) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = static_cast<unsigned>(cluster);
        attr[n].val.clusterDim.y = 1;
        attr[n].val.clusterDim.z = 1;
        ++n;
    }
    if (dependent) {  // may start before the previous kernel on the stream ends (it waits in-kernel)
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    cfg.attrs = n ? attr : nullptr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}
template <typename... KArgs, typename... Args>
inline cudaError_t launch(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                          int cluster, Args&&... args) {
    return launch_ex(false, kernel, grid, block, smem, stream, cluster, static_cast<Args&&>(args)...);
}

}  // namespace osd
