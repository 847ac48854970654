// osd_device.cuh -- device-side building blocks shared by the verify and
// distill kernels: element loads for fp32/bf16, hardware ex2/lg2, online
// (max, sum-exp) merging, mbarrier + bulk-copy wrappers with bounded waits,
// and thread-block-cluster primitives (rank, DSMEM map/load, barriers).
#pragma once

#include <cstdint>
#include <cuda_bf16.h>

namespace osd {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kNegInf = -__builtin_huge_valf();

// ---------------------------------------------------------------- elements
template <typename In> struct Elem;
// Raw 16-byte chunks: max and clamp work on the packed representation.
// kClampBits / kClamp is -1e30 (rounded to the type): below it every logit
// already has probability 0, and clamped entries keep exp() at exactly 0 while
// differences of logits stay finite.
template <> struct Elem<float> {
    static constexpr int kVec = 4;  // elements per 16-byte vector
    __device__ static float max_raw(const uint4& r) {
        return fmaxf(fmaxf(__uint_as_float(r.x), __uint_as_float(r.y)),
                     fmaxf(__uint_as_float(r.z), __uint_as_float(r.w)));
    }
    __device__ static void clamp_raw(uint4& r) {
        r.x = __float_as_uint(fmaxf(__uint_as_float(r.x), -1e30f));
        r.y = __float_as_uint(fmaxf(__uint_as_float(r.y), -1e30f));
        r.z = __float_as_uint(fmaxf(__uint_as_float(r.z), -1e30f));
        r.w = __float_as_uint(fmaxf(__uint_as_float(r.w), -1e30f));
    }
    __device__ static float clamp1(float x) { return fmaxf(x, -1e30f); }
    __device__ static float min_raw(const uint4& r) {
        return fminf(fminf(__uint_as_float(r.x), __uint_as_float(r.y)),
                     fminf(__uint_as_float(r.z), __uint_as_float(r.w)));
    }
    __device__ static float load(const float* p) { return __ldg(p); }
    __device__ static float lds(const float* p) { return *p; }
    __device__ static void store(float* p, float v) { *p = v; }
    __device__ static void unpack(const uint4& r, float* x) {
        x[0] = __uint_as_float(r.x); x[1] = __uint_as_float(r.y);
        x[2] = __uint_as_float(r.z); x[3] = __uint_as_float(r.w);
    }
};
template <> struct Elem<__nv_bfloat16> {
    static constexpr int kVec = 8;
    static constexpr uint32_t kClampBits = 0xF149F149u;  // bf16 pair of -1.0e30
    __device__ static float max_raw(const uint4& r);
    __device__ static float min_raw(const uint4& r);
    __device__ static void clamp_raw(uint4& r);
    __device__ static float clamp1(float x) { return fmaxf(x, __uint_as_float(0xF1490000u)); }
    __device__ static float load(const __nv_bfloat16* p) {
        return __uint_as_float(uint32_t(__ldg(reinterpret_cast<const unsigned short*>(p))) << 16);
    }
    __device__ static float lds(const __nv_bfloat16* p) {
        return __uint_as_float(uint32_t(*reinterpret_cast<const unsigned short*>(p)) << 16);
    }
    __device__ static void store(__nv_bfloat16* p, float v) {  // only for copying exact bf16 values
        *reinterpret_cast<unsigned short*>(p) = (unsigned short)(__float_as_uint(v) >> 16);
    }
    // bf16 -> fp32 is exact: the bf16 bits are the top half of the fp32 bits.
    __device__ static void unpack(const uint4& r, float* x) {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            x[2 * i] = __uint_as_float(w[i] << 16);
            x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    }
};

// 16-byte streaming global load that bypasses L1 (read-once data).
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(p));
    return r;
}
__device__ __forceinline__ uint4 lds_v4(const void* p) {
    return *reinterpret_cast<const uint4*>(p);
}
__device__ __forceinline__ void stg_v4(float* p, float a, float b, float c, float d) {
    asm volatile("st.global.v4.f32 [%0], {%1,%2,%3,%4};" :: "l"(p), "f"(a), "f"(b), "f"(c), "f"(d)
                 : "memory");
}

// ---------------------------------------------------------------- math
// Hardware base-2 exponential / logarithm (PTX ex2.approx / lg2.approx).
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float lg2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// d * c with c = c_hi + c_lo held as a pair of floats: removes the rounding of
// log2(e)/T from every exponent argument (it would otherwise bias all terms).
__device__ __forceinline__ float mul_c(float d, float c_hi, float c_lo) {
    return fmaf(d, c_hi, d * c_lo);
}

// The two bf16 halves (low = lower address) of a 32-bit word minus m: each half
// converts to fp32 exactly and the difference is rounded once, as unpacking and
// subtracting would give, by the mixed-precision subtract of sm_100+.
__device__ __forceinline__ float2 bf16x2_minus(uint32_t w, float m) {
    float a, b;
    asm("{\n .reg .b16 lo, hi;\n mov.b32 {lo, hi}, %2;\n"
        " sub.rn.f32.bf16 %0, lo, %3;\n sub.rn.f32.bf16 %1, hi, %3;\n}"
        : "=f"(a), "=f"(b) : "r"(w), "f"(m));
    return make_float2(a, b);
}

// ---------------------------------------------------------------- packed f32x2 (sm_100+)
// Two fp32 lanes per instruction; the pack/unpack moves vanish in register allocation.
__device__ __forceinline__ unsigned long long pk2(float a, float b) {
    unsigned long long r;
    asm("mov.b64 %0, {%1,%2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ float2 upk2(unsigned long long r) {
    float2 v;
    asm("mov.b64 {%0,%1}, %2;" : "=f"(v.x), "=f"(v.y) : "l"(r));
    return v;
}
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    unsigned long long d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(pk2(a.x, a.y)), "l"(pk2(b.x, b.y)), "l"(pk2(c.x, c.y)));
    return upk2(d);
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    unsigned long long d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(pk2(a.x, a.y)), "l"(pk2(b.x, b.y)));
    return upk2(d);
}
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
    unsigned long long d;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(pk2(a.x, a.y)), "l"(pk2(b.x, b.y)));
    return upk2(d);
}
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
    unsigned long long d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(pk2(a.x, a.y)), "l"(pk2(b.x, b.y)));
    return upk2(d);
}
__device__ __forceinline__ float2 f2(float a) { return make_float2(a, a); }

// ---------------------------------------------------------------- packed bf16 pairs
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}
__device__ __forceinline__ uint32_t bmin2(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("min.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float Elem<__nv_bfloat16>::max_raw(const uint4& r) {
    const uint32_t m = bmax2(bmax2(r.x, r.y), bmax2(r.z, r.w));
    return fmaxf(bf16_lo(m), bf16_hi(m));
}
__device__ __forceinline__ float Elem<__nv_bfloat16>::min_raw(const uint4& r) {
    const uint32_t m = bmin2(bmin2(r.x, r.y), bmin2(r.z, r.w));
    return fminf(bf16_lo(m), bf16_hi(m));
}
__device__ __forceinline__ void Elem<__nv_bfloat16>::clamp_raw(uint4& r) {
    r.x = bmax2(r.x, kClampBits);
    r.y = bmax2(r.y, kClampBits);
    r.z = bmax2(r.z, kClampBits);
    r.w = bmax2(r.w, kClampBits);
}

// Online softmax statistics of one set of values: m = max, s = sum 2^((x-m)c).
struct MaxSum {
    float m;
    float s;
};
__device__ __forceinline__ MaxSum merge_ms(MaxSum a, MaxSum b, float c_hi, float c_lo) {
    if (b.m > a.m) { MaxSum t = a; a = b; b = t; }
    if (b.m != kNegInf) a.s += b.s * ex2(mul_c(b.m - a.m, c_hi, c_lo));
    return a;
}
// Argmax with the lowest index on ties.
struct MaxIdx {
    float m;
    int i;
};
__device__ __forceinline__ MaxIdx merge_mi(MaxIdx a, MaxIdx b) {
    if (b.m > a.m || (b.m == a.m && b.i < a.i)) return b;
    return a;
}

template <typename T, typename F>
__device__ __forceinline__ T warp_reduce(T v, F f) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        T w;
        if constexpr (sizeof(T) == 8) {
            unsigned long long bits = *reinterpret_cast<unsigned long long*>(&v);
            bits = __shfl_xor_sync(0xffffffffu, bits, o);
            w = *reinterpret_cast<T*>(&bits);
        } else if constexpr (sizeof(T) == 4) {
            unsigned bits = *reinterpret_cast<unsigned*>(&v);
            bits = __shfl_xor_sync(0xffffffffu, bits, o);
            w = *reinterpret_cast<T*>(&bits);
        } else {
            static_assert(sizeof(T) % 4 == 0, "warp_reduce needs 4-byte multiples");
            unsigned* vb = reinterpret_cast<unsigned*>(&v);
            unsigned wb[sizeof(T) / 4];
#pragma unroll
            for (int k = 0; k < int(sizeof(T) / 4); ++k) wb[k] = __shfl_xor_sync(0xffffffffu, vb[k], o);
            w = *reinterpret_cast<T*>(wb);
        }
        v = f(v, w);
    }
    return v;
}

// Block-wide reduction through shared scratch (one slot per warp); result is
// returned to every thread.  `scratch` holds at least kThreads/32 values.
template <int kThreads, typename T, typename F>
__device__ __forceinline__ T block_reduce(T v, F f, T* scratch) {
    constexpr int kWarps = kThreads / 32;
    v = warp_reduce(v, f);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __syncthreads();  // scratch may still be read by a previous reduction
    if (lane == 0) scratch[warp] = v;
    __syncthreads();
    T r = scratch[0];
#pragma unroll
    for (int w = 1; w < kWarps; ++w) r = f(r, scratch[w]);
    return r;
}

// fp64 inclusive prefix sum across a warp (the mixed sampler's CDF scans)
__device__ __forceinline__ double warp_incl_scan_f64(double v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}

// ---------------------------------------------------------------- programmatic dependent launch
// A kernel lets the next kernel on its stream (launched with programmatic stream
// serialisation) start; that kernel waits for this one's results and memory only
// where it calls grid_dependency_wait.  Both are no-ops without the attribute.
__device__ __forceinline__ void allow_dependent_launch() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void grid_dependency_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ---------------------------------------------------------------- timers / errors
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---------------------------------------------------------------- mbarrier + bulk copy
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(smem_addr(bar)), "r"(count) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_init_only(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbarrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
                 :: "r"(smem_addr(bar)), "r"(bytes) : "memory");
}
// One-dimensional bulk copy global -> this CTA's shared memory, completing
// `bytes` transactions on `bar`.  dst, src 16-byte aligned; bytes % 16 == 0.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        :: "r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok) : "r"(smem_addr(bar)), "r"(parity) : "memory");
    return ok != 0;
}
// Arrive on a barrier of this CTA (release at CTA scope: this thread's earlier
// shared-memory writes are visible to the threads that then see the phase end).
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(smem_addr(bar)) : "memory");
}
// The phase test with acquire at cluster scope: for barriers completed by
// st.async writes from other CTAs of the cluster.
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok) : "r"(smem_addr(bar)), "r"(parity) : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_cluster_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    while (!mbar_try_wait_cluster(bar, parity)) {
        if (global_ns() - t0 > limit_ns) return false;
    }
    return true;
}
// 16 bytes into the shared memory of a CTA of the cluster (addr and bar from
// mapa), completing 16 transaction bytes on that CTA's barrier `bar`.
__device__ __forceinline__ void st_async_v4(uint32_t addr, float4 v, uint32_t bar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];"
                 :: "r"(addr), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(bar) : "memory");
}
__device__ __forceinline__ void st_async_v2(uint32_t addr, float2 v, uint32_t bar) {  // 8 bytes
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];"
                 :: "r"(addr), "f"(v.x), "f"(v.y), "r"(bar) : "memory");
}
__device__ __forceinline__ void st_async_u64(uint32_t addr, unsigned long long v, uint32_t bar) {  // 8 bytes
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b64 [%0], %1, [%2];"
                 :: "r"(addr), "l"(v), "r"(bar) : "memory");
}
// Wait for phase `parity` of `bar`, giving up after `limit_ns` of wall time.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (global_ns() - t0 > limit_ns) return false;
    }
    return true;
}

// ---------------------------------------------------------------- clusters
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// The .aligned forms need a converged warp, hence the __syncwarp() first.
// Arrive without ordering: used once this CTA has consumed every value it read
// from its peers' shared memory, to tell them they may exit.
__device__ __forceinline__ void cluster_arrive_relaxed() {
    __syncwarp();
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
// Cluster barrier that publishes shared-memory writes made by the calling
// threads with `writer` set: only they fence, everyone else arrives relaxed,
// and the wait acquires, so the peers see those writes afterwards.
__device__ __forceinline__ void cluster_sync_publish(bool writer) {
    if (writer) asm volatile("fence.acq_rel.cluster;" ::: "memory");
    __syncwarp();
    asm volatile("barrier.cluster.arrive.relaxed.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    __syncwarp();
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of `p` (in this CTA's shared memory) inside CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_rank(const void* p, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
    return r;
}
__device__ __forceinline__ float ld_dsmem_f32(uint32_t addr) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ unsigned long long ld_dsmem_u64(uint32_t addr) {
    unsigned long long v;
    asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ float4 ld_dsmem_v4f32(uint32_t addr) {  // 16-byte aligned
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ float2 ld_dsmem_v2f32(uint32_t addr) {  // 8-byte aligned
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ int ld_dsmem_s32(uint32_t addr) {
    int v;
    asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}

// ---------------------------------------------------------------- tensor memory (tcgen05)
// Tensor memory: 128 lanes x 512 columns of 32-bit cells per SM.  A CTA allocates
// a power-of-two number of columns (32..512) with one warp; warp w of a CTA may
// access lanes 32 (w % 4) .. 32 (w % 4) + 31, each thread its own lane.  An
// address is (lane << 16) | column.
__device__ __forceinline__ void tm_alloc(uint32_t* dst_smem, uint32_t ncols) {  // one whole warp
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 :: "r"(smem_addr(dst_smem)), "r"(ncols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tm_dealloc(uint32_t taddr, uint32_t ncols) {  // one whole warp
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" :: "r"(taddr), "r"(ncols) : "memory");
}
// Order tensor-memory accesses around a thread barrier (alloc -> use -> dealloc).
__device__ __forceinline__ void tm_fence_before_sync() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tm_fence_after_sync() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Eight consecutive columns of this thread's lane (warp-collective, uniform address).
__device__ __forceinline__ void tm_ld8(uint32_t taddr, uint4& a, uint4& b) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w), "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
                 : "r"(taddr) : "memory");
}
__device__ __forceinline__ void tm_ld4(uint32_t taddr, uint4& a) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w) : "r"(taddr) : "memory");
}
__device__ __forceinline__ void tm_st8(uint32_t taddr, const uint4& a, const uint4& b) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};"
                 :: "r"(taddr), "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b.x), "r"(b.y), "r"(b.z), "r"(b.w)
                 : "memory");
}
__device__ __forceinline__ void tm_st4(uint32_t taddr, const uint4& a) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};"
                 :: "r"(taddr), "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w) : "memory");
}
__device__ __forceinline__ void tm_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tm_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// Generic-proxy accesses of shared memory before this point are ordered before
// later async-proxy (bulk copy) writes to it.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Sentinel for vector slots past the end of a row or slice: -inf never
// raises a maximum and adds 0 to a sum.
template <typename In> struct NegInfRaw;
template <> struct NegInfRaw<float> { static constexpr uint32_t bits = 0xFF800000u; };
template <> struct NegInfRaw<__nv_bfloat16> { static constexpr uint32_t bits = 0xFF80FF80u; };

template <typename In> __device__ __forceinline__ uint4 ninf_raw() {
    return make_uint4(NegInfRaw<In>::bits, NegInfRaw<In>::bits, NegInfRaw<In>::bits, NegInfRaw<In>::bits);
}
// kW values of type In held in (the low bytes of) a 16-byte register block.
template <typename In, int kW>
__device__ __forceinline__ uint4 pack_raw(const float* v) {
    if constexpr (kW == 1) {
        return make_uint4(__float_as_uint(v[0]), 0u, 0u, 0u);
    } else if constexpr (sizeof(In) == 4) {
        return make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]), __float_as_uint(v[3]));
    } else {  // bf16: the values are exact bf16 numbers, so truncation keeps them
        uint32_t w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) w[i] = (__float_as_uint(v[2 * i]) >> 16) | (__float_as_uint(v[2 * i + 1]) & 0xffff0000u);
        return make_uint4(w[0], w[1], w[2], w[3]);
    }
}
template <typename In, int kW>
__device__ __forceinline__ void unpack_raw(const uint4& r, float* v) {
    if constexpr (kW == 1) v[0] = __uint_as_float(r.x);
    else Elem<In>::unpack(r, v);
}

// ---------------------------------------------------------------- exact CDF sums
// Non-negative weights below 8 as unsigned 64-bit fixed point with kFixBits
// fraction bits, truncated.  Sums of them are exact, so a prefix sum does not
// depend on the order of its adds; and an integer add takes a few cycles where
// a dependent fp64 add takes about 64 on this GPU.  Truncation loses less than
// 2^-60 per weight.
constexpr int kFixBits = 60;
__device__ __forceinline__ unsigned long long fix_of(float x) {
    const uint32_t bits = __float_as_uint(x);
    const int e = static_cast<int>(bits >> 23);  // x >= 0: no sign bit
    if (e == 0) return 0ull;                     // zero or subnormal, below 2^-126
    const unsigned long long m = (bits & 0x7fffffu) | 0x800000u;
    const int sh = e - (127 + 23) + kFixBits;    // x = m 2^(e - 150)
    return sh >= 0 ? (m << sh) : (sh > -64 ? (m >> -sh) : 0ull);
}
__device__ __forceinline__ float fix_to_float(unsigned long long v) {
    return __ull2float_rn(v) * (1.0f / static_cast<float>(1ull << kFixBits));
}
// floor(u W) for u in [0, 1) (u >= 1 gives W): u as a 64-bit binary fraction,
// exact for u >= 2^-40, times W, high half.
__device__ __forceinline__ unsigned long long fix_scale(float u, unsigned long long W) {
    const uint32_t bits = __float_as_uint(u);
    const int e = static_cast<int>(bits >> 23);
    if (e == 0 || (bits >> 31)) return 0ull;
    if (e >= 127) return W;
    const unsigned long long m = (bits & 0x7fffffu) | 0x800000u;
    const int sh = e - 150 + 64;  // <= 40 for u < 1
    const unsigned long long U = sh >= 0 ? (m << sh) : (sh > -64 ? (m >> -sh) : 0ull);
    return __umul64hi(U, W);
}
__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ unsigned long long warp_incl_scan_u64(unsigned long long v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}

}  // namespace osd
