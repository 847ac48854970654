// osd_rowspan.cuh -- building blocks of the kernels that stage one span of a
// draft row and a target row in shared memory and sweep it several times
// (distillation and mixed sampling).  One thread-block cluster per row, each
// CTA of kRowThreads (or a template's kT) threads owns a contiguous span of the
// vocabulary.
#pragma once

#include <cstddef>
#include <cstdint>
#include <type_traits>

#include "osd_device.cuh"

namespace osd {

constexpr int kRowThreads = 128;
constexpr int kRowWarps = kRowThreads / 32;
constexpr uint64_t kStageWaitNs = 1000000000ull;  // bound on the wait for the bulk copies

template <typename In>
__device__ __forceinline__ void copy_raw(In* dst, const In* src) {
    using Raw = std::conditional_t<sizeof(In) == 2, unsigned short, unsigned int>;
    *reinterpret_cast<Raw*>(dst) = __ldg(reinterpret_cast<const Raw*>(src));
}

// Stage n entries of a draft and a target row (zsrc, tsrc) into zs, ts.  On the
// aligned path the 16-byte body goes by two bulk copies completing on `bar`
// and the ragged tail by plain loads.  Every thread calls it; it returns
// non-zero (for every thread) when the bounded wait for the copies gave up.
template <typename In, bool kAligned, int kT = kRowThreads>
__device__ __forceinline__ int stage_span(In* zs, In* ts, const In* zsrc, const In* tsrc, int n, uint64_t* bar,
                                          int* s_err) {
    const int tid = threadIdx.x;
    if (tid == 0) *s_err = 0;
    if constexpr (kAligned) {
        const uint32_t bytes = static_cast<uint32_t>(n * sizeof(In)) & ~15u;
        const int nb = static_cast<int>(bytes / sizeof(In));
        if (tid == 0 && bytes) mbar_init(bar, 1);
        __syncthreads();
        if (tid == 0 && bytes) {
            mbar_arrive_expect_tx(bar, 2 * bytes);
            bulk_g2s(zs, zsrc, bytes, bar);
            bulk_g2s(ts, tsrc, bytes, bar);
        }
        for (int e = nb + tid; e < n; e += kT) {
            copy_raw(zs + e, zsrc + e);
            copy_raw(ts + e, tsrc + e);
        }
        if (bytes && !mbar_wait_bounded(bar, 0, kStageWaitNs)) {
            atomicOr(s_err, 1);
            mbar_wait_bounded(bar, 0, kStageWaitNs);  // give copies in flight a last chance to land
        }
    } else {
        __syncthreads();
        for (int e = tid; e < n; e += kT) {
            copy_raw(zs + e, zsrc + e);
            copy_raw(ts + e, tsrc + e);
        }
    }
    __syncthreads();
    return *s_err;
}

// stage_span in two halves, for a caller with other work to do while the copies
// fly: stage_span_issue (thread 0 initialises `bar` and issues the bulk copies;
// a block barrier must come before any other thread waits on `bar`), then
// stage_span_land (the ragged tail by plain loads, the bounded wait, a block
// barrier; returns non-zero, for every thread, when the wait gave up).
template <typename In, bool kAligned>
__device__ __forceinline__ void stage_span_issue(In* zs, In* ts, const In* zsrc, const In* tsrc, int n,
                                                 uint64_t* bar, int* s_err) {
    if (threadIdx.x == 0) *s_err = 0;
    if constexpr (kAligned) {
        const uint32_t bytes = static_cast<uint32_t>(n * sizeof(In)) & ~15u;
        if (threadIdx.x == 0 && bytes) {
            mbar_init(bar, 1);
            mbar_arrive_expect_tx(bar, 2 * bytes);
            bulk_g2s(zs, zsrc, bytes, bar);
            bulk_g2s(ts, tsrc, bytes, bar);
        }
    }
}
template <typename In, bool kAligned, int kT = kRowThreads>
__device__ __forceinline__ int stage_span_land(In* zs, In* ts, const In* zsrc, const In* tsrc, int n, uint64_t* bar,
                                               int* s_err) {
    const int tid = threadIdx.x;
    const uint32_t bytes = kAligned ? (static_cast<uint32_t>(n * sizeof(In)) & ~15u) : 0u;
    const int nb = static_cast<int>(bytes / sizeof(In));
    for (int e = nb + tid; e < n; e += kT) {
        copy_raw(zs + e, zsrc + e);
        copy_raw(ts + e, tsrc + e);
    }
    if (bytes && !mbar_wait_bounded(bar, 0, kStageWaitNs)) {
        atomicOr(s_err, 1);
        mbar_wait_bounded(bar, 0, kStageWaitNs);  // give copies in flight a last chance to land
    }
    __syncthreads();
    return *s_err;
}

// Visit this thread's entries of a staged span in chunks of one 16-byte vector
// (or single entries on the element-wise path).  Clamping (to -1e30, see Elem)
// happens on the packed words.  f(z[], t[], count_tag, j0, zmax, tmax, ninf,
// zraw, traw) gets the chunk maxima when kMax is set, ninf = "the chunk holds a
// -inf" when kMin is set, and the (clamped) packed words of a full chunk.
// Chunk v goes to thread v mod kT (the CTA's threads), so warp w sees the
// 32-chunk groups w, w + kT/32, ... in order.  kUnroll unrolls the chunk loop
// (two chunks a trip halve the loop overhead, at some registers).
template <typename In, bool kAligned, bool kClampZ, bool kClampT, bool kMax, bool kMin = false, int kUnroll = 1,
          int kT = kRowThreads, typename F>
__device__ __forceinline__ void sweep(const In* zs, const In* ts, int n, F&& f) {
    using E = Elem<In>;
    constexpr int kVec = E::kVec;
    const int tid = threadIdx.x;
    if constexpr (kAligned) {
        const int nv = n / kVec;
#pragma unroll kUnroll
        for (int v = tid; v < nv; v += kT) {
            uint4 zr = lds_v4(zs + v * kVec), tr = lds_v4(ts + v * kVec);
            if (kClampZ) E::clamp_raw(zr);
            if (kClampT) E::clamp_raw(tr);
            float z[kVec], t[kVec];
            E::unpack(zr, z);
            E::unpack(tr, t);
            const float cz = kMax ? E::max_raw(zr) : 0.f, ct = kMax ? E::max_raw(tr) : 0.f;
            const bool ninf = kMin ? (fminf(E::min_raw(zr), E::min_raw(tr)) == kNegInf) : false;
            f(z, t, std::integral_constant<int, kVec>{}, v * kVec, cz, ct, ninf, zr, tr);
        }
        const int r0 = nv * kVec;
        if (tid < n - r0) {
            float z = E::lds(zs + r0 + tid), t = E::lds(ts + r0 + tid);
            if (kClampZ) z = E::clamp1(z);
            if (kClampT) t = E::clamp1(t);
            f(&z, &t, std::integral_constant<int, 1>{}, r0 + tid, z, t, fminf(z, t) == kNegInf, uint4{}, uint4{});
        }
    } else {
        for (int e = tid; e < n; e += kT) {
            float z = E::lds(zs + e), t = E::lds(ts + e);
            if (kClampZ) z = E::clamp1(z);
            if (kClampT) t = E::clamp1(t);
            f(&z, &t, std::integral_constant<int, 1>{}, e, z, t, fminf(z, t) == kNegInf, uint4{}, uint4{});
        }
    }
}

// Block-wide max of two values, then sum of three: the cheap way to merge
// softmax partials (every thread rescales its sums once to the block max).
// kGuard adds the barrier that keeps a previous reduction's readers of
// `scratch` ahead of the new writes; callers whose scratch has no readers
// since the last block barrier leave it out.
template <bool kGuard = true, int kT = kRowThreads>
__device__ __forceinline__ float2 block_max2(float a, float b, float2* scratch) {
    for (int o = 16; o > 0; o >>= 1) {
        a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
        b = fmaxf(b, __shfl_xor_sync(0xffffffffu, b, o));
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (kGuard) __syncthreads();
    if (lane == 0) scratch[warp] = make_float2(a, b);
    __syncthreads();
    float2 r = scratch[0];
#pragma unroll
    for (int w = 1; w < kT / 32; ++w) r = make_float2(fmaxf(r.x, scratch[w].x), fmaxf(r.y, scratch[w].y));
    return r;
}
template <bool kGuard = true, int kT = kRowThreads>
__device__ __forceinline__ float3 block_sum3(float a, float b, float c, float3* scratch) {
    for (int o = 16; o > 0; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o);
        b += __shfl_xor_sync(0xffffffffu, b, o);
        c += __shfl_xor_sync(0xffffffffu, c, o);
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (kGuard) __syncthreads();
    if (lane == 0) scratch[warp] = make_float3(a, b, c);
    __syncthreads();
    float3 r = scratch[0];
#pragma unroll
    for (int w = 1; w < kT / 32; ++w) r = make_float3(r.x + scratch[w].x, r.y + scratch[w].y, r.z + scratch[w].z);
    return r;
}

// Split V over a cluster: about span_bytes of staged logits (both rows) per
// CTA, at most max_cluster CTAs, spans a multiple of 64 entries, at most
// max_smem bytes of staging per CTA.  Returns false when V does not fit.
inline bool row_span_shape(int V, size_t es, size_t span_bytes, int max_cluster, size_t max_smem, int* csize,
                           int* span) {
    const int base = static_cast<int>(span_bytes / (2 * es));
    int c = (V + base - 1) / base;
    if (c > max_cluster) c = max_cluster;
    if (c < 1) c = 1;
    int s = (V + c - 1) / c;
    s = (s + 63) / 64 * 64;
    c = (V + s - 1) / s;
    if (2 * size_t(s) * es > max_smem) return false;
    *csize = c;
    *span = s;
    return true;
}

}  // namespace osd
