// osd_distill.cu -- per-position distillation loss and gradient (Eq. 2-3 of
// the paper, Section 4.1; the analytic draft update of Algorithm 1) on sm_103a.
//
// One thread-block cluster per active row.  Each CTA owns a contiguous span of
// the vocabulary: it stages its span of the draft and target rows into shared
// memory with two bulk copies (cp.async.bulk, completion on an mbarrier), so
// each logit is read from HBM exactly once.  The row never leaves the chip:
//
//   pass 1  online max / sum-exp of both rows (+ the loss moment of FKL/RKL),
//           merged across the cluster through distributed shared memory;
//   pass 2  (JSD, TVD only) the per-entry divergence terms, which need the
//           global normalisers, merged the same way;
//   pass 3  d loss / d draft logits for the span, written with 16-byte stores.
//
// Every CTA merges the cluster's partials in rank order, so all CTAs of a row
// see bit-identical statistics.  Logs and exponentials use the hardware
// lg2/ex2 units in base 2; loss terms are converted to nats at the end.
#include <climits>
#include <cstdint>
#include <type_traits>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"

namespace osd {

constexpr int kDistThreads = 256;
constexpr int kDistMaxCluster = 8;
constexpr int kDistSpanBytes = 32768;         // target bytes of both rows per CTA
constexpr int kDistMaxSmem = 192 * 1024;      // largest staging buffer per CTA
constexpr uint64_t kWaitLimitNs = 1000000000ull;

struct DistParams {
    const void* draft;
    const void* target;
    int G, P, V;
    long long dsg, dsp, tsg, tsp;
    const uint8_t* mask;
    float beta;
    float* loss;
    float* dlogits;
    int32_t* status;
    int csize;  // CTAs per row (cluster size)
    int span;   // vocabulary entries per CTA (multiple of 64)
};

// Pass-1 partial of a span: maxima, sums of 2^((x-m) log2 e) and one loss moment.
struct Stats1 {
    float mz, Ez, mt, Et, X;
    int err;
};
// Pass-2 partial: JSD (KL(p||m), KL(q||m)) in bits, or TVD (sum |p-q|, sum q g).
struct Stats2 {
    float a, b;
};

template <int kKind>
__device__ __forceinline__ Stats1 merge1(Stats1 a, Stats1 b) {
    Stats1 r;
    r.mz = fmaxf(a.mz, b.mz);
    r.mt = fmaxf(a.mt, b.mt);
    const float az = (a.mz == kNegInf) ? 0.f : ex2((a.mz - r.mz) * kLog2e);
    const float bz = (b.mz == kNegInf) ? 0.f : ex2((b.mz - r.mz) * kLog2e);
    const float at = (a.mt == kNegInf) ? 0.f : ex2((a.mt - r.mt) * kLog2e);
    const float bt = (b.mt == kNegInf) ? 0.f : ex2((b.mt - r.mt) * kLog2e);
    r.Ez = a.Ez * az + b.Ez * bz;
    r.Et = a.Et * at + b.Et * bt;
    if (kKind == OSD_FKL) r.X = a.X * at + b.X * bt;       // weighted by target exponentials
    else if (kKind == OSD_RKL) r.X = a.X * az + b.X * bz;  // weighted by draft exponentials
    else r.X = 0.f;
    r.err = a.err | b.err;
    return r;
}

// log2 of a probability, (x - m) log2(e) - log2(s), with every operation rounded
// on its own: the draft and target sides, and passes 2 and 3, must round alike so
// that sign(q - p) is exactly 0 where the two rows agree.
__device__ __forceinline__ float log2_prob(float x, float m, float l2s) {
    return __fsub_rn(__fmul_rn(__fsub_rn(x, m), kLog2e), l2s);
}

template <typename In>
__device__ __forceinline__ void copy_raw(In* dst, const In* src) {
    using Raw = std::conditional_t<sizeof(In) == 2, unsigned short, unsigned int>;
    *reinterpret_cast<Raw*>(dst) = __ldg(reinterpret_cast<const Raw*>(src));
}

// Visit this thread's entries of a staged span: f(z[], t[], count_tag, j0).
template <typename In, bool kAligned, typename F>
__device__ __forceinline__ void sweep(const In* zs, const In* ts, int n, F&& f) {
    using E = Elem<In>;
    constexpr int kVec = E::kVec;
    const int tid = threadIdx.x;
    if constexpr (kAligned) {
        const int nv = n / kVec;
        for (int v = tid; v < nv; v += kDistThreads) {
            float z[kVec], t[kVec];
            E::unpack(lds_v4(zs + v * kVec), z);
            E::unpack(lds_v4(ts + v * kVec), t);
            f(z, t, std::integral_constant<int, kVec>{}, v * kVec);
        }
        const int r0 = nv * kVec;
        if (tid < n - r0) {
            const float z = E::lds(zs + r0 + tid), t = E::lds(ts + r0 + tid);
            f(&z, &t, std::integral_constant<int, 1>{}, r0 + tid);
        }
    } else {
        for (int e = tid; e < n; e += kDistThreads) {
            const float z = E::lds(zs + e), t = E::lds(ts + e);
            f(&z, &t, std::integral_constant<int, 1>{}, e);
        }
    }
}

template <typename In, int kKind, bool kAligned>
__global__ void __launch_bounds__(kDistThreads) distill_kernel(DistParams p) {
    using E = Elem<In>;
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ Stats1 s1_mine, s1_all;
    __shared__ Stats2 s2_mine, s2_all;
    __shared__ Stats1 red1[kDistThreads / 32];
    __shared__ Stats2 red2[kDistThreads / 32];
    __shared__ int s_err;

    const int tid = threadIdx.x;
    const int csize = p.csize;
    const int rank = (csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    const long long row = blockIdx.x / csize;
    if (p.mask && !p.mask[row]) {  // uniform over the cluster; no shared memory is exchanged
        if (rank == 0 && tid == 0) p.loss[row] = 0.f;
        return;
    }
    const long long g = row / p.P, pp = row - g * p.P;
    const In* zrow = static_cast<const In*>(p.draft) + g * p.dsg + pp * p.dsp;
    const In* trow = static_cast<const In*>(p.target) + g * p.tsg + pp * p.tsp;
    const int V = p.V;
    const int e0 = rank * p.span;
    const int n = min(p.span, V - e0);
    In* zs = reinterpret_cast<In*>(dsm);
    In* ts = zs + p.span;

    // ---- stage the span of both rows in shared memory
    if (tid == 0) s_err = 0;
    bool ok = true;
    if constexpr (kAligned) {
        const uint32_t bytes = static_cast<uint32_t>(n * sizeof(In)) & ~15u;
        const int nb = static_cast<int>(bytes / sizeof(In));
        if (tid == 0 && bytes) mbar_init(&bar, 1);
        __syncthreads();
        if (tid == 0 && bytes) {
            mbar_arrive_expect_tx(&bar, 2 * bytes);
            bulk_g2s(zs, zrow + e0, bytes, &bar);
            bulk_g2s(ts, trow + e0, bytes, &bar);
        }
        for (int e = nb + tid; e < n; e += kDistThreads) {
            copy_raw(zs + e, zrow + e0 + e);
            copy_raw(ts + e, trow + e0 + e);
        }
        if (bytes) {
            ok = mbar_wait_bounded(&bar, 0, kWaitLimitNs);
            if (!ok) {
                atomicOr(&s_err, 1);
                mbar_wait_bounded(&bar, 0, kWaitLimitNs);  // give copies in flight a last chance to land
            }
        }
    } else {
        __syncthreads();
        for (int e = tid; e < n; e += kDistThreads) {
            copy_raw(zs + e, zrow + e0 + e);
            copy_raw(ts + e, trow + e0 + e);
        }
    }
    __syncthreads();
    const int err_local = s_err;

    // ---- pass 1: online max / sum-exp (+ loss moment) of the span
    Stats1 acc{kNegInf, 0.f, kNegInf, 0.f, 0.f, err_local};
    if (!err_local) {
        sweep<In, kAligned>(zs, ts, n, [&](const float* z, const float* t, auto tag, int) {
            constexpr int kCnt = decltype(tag)::value;
            float cz = z[0], ct = t[0];
#pragma unroll
            for (int e = 1; e < kCnt; ++e) { cz = fmaxf(cz, z[e]); ct = fmaxf(ct, t[e]); }
            if (cz > acc.mz) {
                const float r = (acc.mz == kNegInf) ? 0.f : ex2((acc.mz - cz) * kLog2e);
                acc.Ez *= r;
                if (kKind == OSD_RKL) acc.X *= r;
                acc.mz = cz;
            }
            if (ct > acc.mt) {
                const float r = (acc.mt == kNegInf) ? 0.f : ex2((acc.mt - ct) * kLog2e);
                acc.Et *= r;
                if (kKind == OSD_FKL) acc.X *= r;
                acc.mt = ct;
            }
            if (acc.mz != kNegInf) {
#pragma unroll
                for (int e = 0; e < kCnt; ++e) {
                    const float ez = ex2((z[e] - acc.mz) * kLog2e);
                    acc.Ez += ez;
                    if (kKind == OSD_RKL) acc.X += (ez > 0.f) ? ez * (z[e] - t[e]) : 0.f;
                }
            }
            if (acc.mt != kNegInf) {
#pragma unroll
                for (int e = 0; e < kCnt; ++e) {
                    const float et = ex2((t[e] - acc.mt) * kLog2e);
                    acc.Et += et;
                    if (kKind == OSD_FKL) acc.X += (et > 0.f) ? et * (t[e] - z[e]) : 0.f;
                }
            }
        });
    }
    acc = block_reduce<kDistThreads>(acc, [](Stats1 a, Stats1 b) { return merge1<kKind>(a, b); }, red1);
    if (tid == 0) s1_mine = acc;
    if (csize > 1) cluster_sync(); else __syncthreads();
    if (tid == 0) {
        Stats1 all = s1_mine;
        if (csize > 1) {
            for (int r = 0; r < csize; ++r) {
                Stats1 o;
                if (r == rank) {
                    o = s1_mine;
                } else {
                    const uint32_t base = map_rank(&s1_mine, r);
                    o.mz = ld_dsmem_f32(base + offsetof(Stats1, mz));
                    o.Ez = ld_dsmem_f32(base + offsetof(Stats1, Ez));
                    o.mt = ld_dsmem_f32(base + offsetof(Stats1, mt));
                    o.Et = ld_dsmem_f32(base + offsetof(Stats1, Et));
                    o.X = ld_dsmem_f32(base + offsetof(Stats1, X));
                    o.err = ld_dsmem_s32(base + offsetof(Stats1, err));
                }
                all = (r == 0) ? o : merge1<kKind>(all, o);
            }
        }
        s1_all = all;
    }
    __syncthreads();
    const Stats1 st = s1_all;
    const bool row_err = st.err != 0;
    const float invEz = 1.0f / st.Ez, invEt = 1.0f / st.Et;
    float loss = 0.f;
    if (kKind == OSD_FKL) loss = st.X * invEt - (st.mt - st.mz) - logf(st.Et * invEz);
    if (kKind == OSD_RKL) loss = st.X * invEz - (st.mz - st.mt) - logf(st.Ez * invEt);

    const float beta = p.beta;
    const bool jsd_trivial = (kKind == OSD_JSD) && (beta == 0.f || beta == 1.f);  // m = q or m = p: loss 0
    const float l2Ez = log2f(st.Ez), l2Et = log2f(st.Et);
    Stats2 s2 = {0.f, 0.f};
    if constexpr (kKind == OSD_JSD || kKind == OSD_TVD) {
        // ---- pass 2: divergence terms with the global normalisers
        Stats2 a2{0.f, 0.f};
        if (!row_err && !jsd_trivial) {
            sweep<In, kAligned>(zs, ts, n, [&](const float* z, const float* t, auto tag, int) {
                constexpr int kCnt = decltype(tag)::value;
#pragma unroll
                for (int e = 0; e < kCnt; ++e) {
                    const float u = log2_prob(t[e], st.mt, l2Et);  // log2 p
                    const float v = log2_prob(z[e], st.mz, l2Ez);  // log2 q
                    const float d = v - u;
                    if (kKind == OSD_TVD) {
                        const float pj = ex2(u), qj = ex2(v);
                        a2.a += fabsf(pj - qj);
                        a2.b += qj * ((d > 0.f) ? 0.5f : ((d < 0.f) ? -0.5f : 0.f));
                    } else {
                        const float ad = fabsf(d);
                        const float big = ex2(fmaxf(u, v));
                        const float rho = ex2(-ad);  // smaller / larger of p, q
                        const bool pbig = d <= 0.f;
                        const float pj = pbig ? big : big * rho;
                        const float qj = pbig ? big * rho : big;
                        const float wbig = pbig ? beta : 1.f - beta;
                        const float L = lg2(wbig + (1.f - wbig) * rho);  // log2(m / larger)
                        const float l2mp = pbig ? L : L + ad;
                        const float l2mq = pbig ? L + ad : L;
                        a2.a += (pj > 0.f) ? -pj * l2mp : 0.f;
                        a2.b += (qj > 0.f) ? -qj * l2mq : 0.f;
                    }
                }
            });
        }
        a2 = block_reduce<kDistThreads>(a2, [](Stats2 x, Stats2 y) { return Stats2{x.a + y.a, x.b + y.b}; }, red2);
        if (tid == 0) s2_mine = a2;
        if (csize > 1) cluster_sync(); else __syncthreads();
        if (tid == 0) {
            Stats2 all{0.f, 0.f};
            for (int r = 0; r < csize; ++r) {
                Stats2 o;
                if (r == rank) {
                    o = s2_mine;
                } else {
                    const uint32_t base = map_rank(&s2_mine, r);
                    o.a = ld_dsmem_f32(base + offsetof(Stats2, a));
                    o.b = ld_dsmem_f32(base + offsetof(Stats2, b));
                }
                all.a += o.a;
                all.b += o.b;
            }
            s2_all = all;
        }
        __syncthreads();
        s2 = s2_all;
        if (kKind == OSD_TVD) loss = 0.5f * s2.a;
        else loss = jsd_trivial ? 0.f : kLn2 * (beta * s2.a + (1.f - beta) * s2.b);
    }
    if (csize > 1) cluster_arrive();  // finished reading the other CTAs' shared memory

    if (rank == 0 && tid == 0) {
        p.loss[row] = row_err ? __int_as_float(0x7fc00000) : loss;
        if (row_err && p.status) atomicExch(p.status, static_cast<int32_t>(OSD_ERR_TIMEOUT));
    }

    // ---- pass 3: d loss / d draft logits of the span
    if (!row_err) {
        float* orow = p.dlogits + row * V + e0;
        const float K_rkl = (st.mz - st.mt) + logf(st.Ez * invEt) + loss;  // RKL: lq - lp - loss = (z - t) - K
        const float jsd_scale = (1.f - beta) * kLn2;
        sweep<In, kAligned>(zs, ts, n, [&](const float* z, const float* t, auto tag, int j0) {
            constexpr int kCnt = decltype(tag)::value;
            float gr[kCnt];
#pragma unroll
            for (int e = 0; e < kCnt; ++e) {
                const float qj = ex2((z[e] - st.mz) * kLog2e) * invEz;
                if (kKind == OSD_FKL) {
                    gr[e] = qj - ex2((t[e] - st.mt) * kLog2e) * invEt;
                } else if (kKind == OSD_RKL) {
                    gr[e] = (qj > 0.f) ? qj * ((z[e] - t[e]) - K_rkl) : 0.f;
                } else if (kKind == OSD_TVD) {
                    const float d = log2_prob(z[e], st.mz, l2Ez) - log2_prob(t[e], st.mt, l2Et);
                    const float sg = (d > 0.f) ? 0.5f : ((d < 0.f) ? -0.5f : 0.f);
                    gr[e] = qj * (sg - s2.b);
                } else {
                    if (jsd_trivial) {
                        gr[e] = 0.f;
                    } else {
                        const float u = log2_prob(t[e], st.mt, l2Et);
                        const float v = log2_prob(z[e], st.mz, l2Ez);
                        const float d = v - u, ad = fabsf(d);
                        const float rho = ex2(-ad);
                        const bool pbig = d <= 0.f;
                        const float wbig = pbig ? beta : 1.f - beta;
                        const float L = lg2(wbig + (1.f - wbig) * rho);
                        const float l2mq = pbig ? L + ad : L;
                        gr[e] = (qj > 0.f) ? jsd_scale * qj * (-l2mq - s2.b) : 0.f;
                    }
                }
            }
            if constexpr (kAligned && kCnt >= 4) {
#pragma unroll
                for (int e = 0; e < kCnt; e += 4) stg_v4(orow + j0 + e, gr[e], gr[e + 1], gr[e + 2], gr[e + 3]);
            } else {
#pragma unroll
                for (int e = 0; e < kCnt; ++e) orow[j0 + e] = gr[e];
            }
        });
    }
    if (csize > 1) cluster_wait();  // keep this CTA's statistics readable until every peer is done
}

// ------------------------------------------------------------------ host
template <typename In, int kKind, bool kAligned>
static cudaError_t launch_distill_kind(const DistParams& dp, long long rows, size_t smem, cudaStream_t s) {
    auto kern = distill_kernel<In, kKind, kAligned>;
    if (smem > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return launch(kern, dim3(static_cast<unsigned>(rows * dp.csize)), dim3(kDistThreads), smem, s,
                  dp.csize, dp);
}

template <typename In, bool kAligned>
static cudaError_t launch_distill_dtype(osd_loss kind, const DistParams& dp, long long rows, size_t smem,
                                        cudaStream_t s) {
    switch (kind) {
        case OSD_FKL: return launch_distill_kind<In, OSD_FKL, kAligned>(dp, rows, smem, s);
        case OSD_RKL: return launch_distill_kind<In, OSD_RKL, kAligned>(dp, rows, smem, s);
        case OSD_JSD: return launch_distill_kind<In, OSD_JSD, kAligned>(dp, rows, smem, s);
        default: return launch_distill_kind<In, OSD_TVD, kAligned>(dp, rows, smem, s);
    }
}

// Split V over a cluster: about kDistSpanBytes of staged logits per CTA, at
// most kDistMaxCluster CTAs, spans a multiple of 64 entries.
static bool distill_shape(int V, size_t es, int* csize, int* span) {
    const int base = static_cast<int>(kDistSpanBytes / (2 * es));
    int c = (V + base - 1) / base;
    if (c > kDistMaxCluster) c = kDistMaxCluster;
    if (c < 1) c = 1;
    int s = (V + c - 1) / c;
    s = (s + 63) / 64 * 64;
    c = (V + s - 1) / s;
    if (2 * size_t(s) * es > size_t(kDistMaxSmem)) return false;
    *csize = c;
    *span = s;
    return true;
}

}  // namespace osd

extern "C" osd_status osd_distill(const void* draft_logits, const void* target_logits, osd_dtype dtype,
                                  int G, int P, int V, int64_t d_stride_g, int64_t d_stride_p,
                                  int64_t t_stride_g, int64_t t_stride_p, const uint8_t* mask, osd_loss kind,
                                  float beta, float* loss, float* dlogits, int32_t* status, void* stream) {
    using namespace osd;
    if (dtype != OSD_F32 && dtype != OSD_BF16) return OSD_ERR_INVALID_ARG;
    if (kind < OSD_FKL || kind > OSD_TVD) return OSD_ERR_INVALID_ARG;
    if (G < 0 || P < 0 || V < 1) return OSD_ERR_INVALID_ARG;
    if (d_stride_g < 0 || d_stride_p < 0 || t_stride_g < 0 || t_stride_p < 0) return OSD_ERR_INVALID_ARG;
    if (kind == OSD_JSD && !(beta >= 0.f && beta <= 1.f)) return OSD_ERR_INVALID_ARG;
    const size_t es = dtype_size(dtype);
    int csize = 1, span = V;
    if (!distill_shape(V, es, &csize, &span)) return OSD_ERR_UNSUPPORTED;
    const long long rows = static_cast<long long>(G) * P;
    if (rows * csize > INT_MAX) return OSD_ERR_UNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (status) {
        if (!aligned_to(status, 4)) return OSD_ERR_INVALID_ARG;
    }
    if (rows == 0) {
        return status ? from_cuda(cudaMemsetAsync(status, 0, sizeof(int32_t), s)) : OSD_OK;
    }
    if (!draft_logits || !target_logits || !loss || !dlogits) return OSD_ERR_INVALID_ARG;
    if (!aligned_to(draft_logits, es) || !aligned_to(target_logits, es) || !aligned_to(loss, 4) ||
        !aligned_to(dlogits, 4))
        return OSD_ERR_INVALID_ARG;
    if (status) {
        const cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
        if (e != cudaSuccess) return OSD_ERR_CUDA;
    }
    auto row_ok = [&](int64_t stride, int count) { return count <= 1 || (stride * int64_t(es)) % 16 == 0; };
    const bool aligned = aligned_to(draft_logits, 16) && aligned_to(target_logits, 16) &&
                         aligned_to(dlogits, 16) && (size_t(V) * 4) % 16 == 0 &&
                         row_ok(d_stride_g, G) && row_ok(d_stride_p, P) && row_ok(t_stride_g, G) &&
                         row_ok(t_stride_p, P);
    DistParams dp;
    dp.draft = draft_logits; dp.target = target_logits;
    dp.G = G; dp.P = P; dp.V = V;
    dp.dsg = d_stride_g; dp.dsp = d_stride_p; dp.tsg = t_stride_g; dp.tsp = t_stride_p;
    dp.mask = mask; dp.beta = beta; dp.loss = loss; dp.dlogits = dlogits; dp.status = status;
    dp.csize = csize; dp.span = span;
    const size_t smem = 2 * size_t(span) * es;
    cudaError_t e;
    if (dtype == OSD_BF16)
        e = aligned ? launch_distill_dtype<__nv_bfloat16, true>(kind, dp, rows, smem, s)
                    : launch_distill_dtype<__nv_bfloat16, false>(kind, dp, rows, smem, s);
    else
        e = aligned ? launch_distill_dtype<float, true>(kind, dp, rows, smem, s)
                    : launch_distill_dtype<float, false>(kind, dp, rows, smem, s);
    return from_cuda(e);
}
