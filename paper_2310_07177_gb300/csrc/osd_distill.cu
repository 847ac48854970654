// osd_distill.cu -- per-position distillation loss and gradient (Eq. 2-3 of
// the paper, Section 4.1, with its softmax temperature; the analytic draft
// update of Algorithm 1; and the label fine-tuning cross-entropy of Table 1)
// on sm_103a.
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
//
// Buffer flushes of 16-byte-aligned rows (FKL, RKL, JSD, TVD) take the
// TMEM-staged runs of rows further down instead, which overlap the copy of a
// row with the passes of the one before it.
#include <algorithm>
#include <atomic>
#include <climits>
#include <cmath>
#include <cstdint>
#include <mutex>
#include <type_traits>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"
#include "osd_rowspan.cuh"

namespace osd {

constexpr int kDistThreads = kRowThreads;      // threads per CTA ...
constexpr int kDistThreadsWide = 256;          // ... and for spans of kDistWideSpan entries or more, where
constexpr int kDistWideSpan = 12288;           // FKL, RKL, CE and JSD measured 5-10 % faster (V = 128256)
constexpr int kDistMaxCluster = 8;            // CTAs per row that bound the vocabulary (V limits) ...
constexpr int kDistMaxClusterWide = 16;       // ... and up to 16 (non-portable clusters) where a row needs
                                              // more than 8 spans of the target size (V > 65536 bf16)
constexpr int kDistSpanBytes = 32768;         // target bytes of both rows per CTA
constexpr int kDistSpanBytesJsd = 49152;      // JSD, with the most work per entry, does best with fewer, longer spans
constexpr int kDistMaxSmem = 192 * 1024;      // largest staging buffer per CTA
constexpr float kMinNormal = 1.17549435e-38f;  // smallest normal fp32

struct DistParams {
    const void* draft;
    const void* target;
    int G, P, V;
    long long dsg, dsp, tsg, tsp;
    const uint8_t* mask;
    float beta;
    float c;        // log2(e) / temperature: exp(x / tau) = 2^(x c)
    float inv_tau;  // the gradient w.r.t. raw logits carries 1 / tau
    float lg_scale; // log2 of the gradient's constant factor (1/tau; JSD (1-beta) ln2 / tau),
                    // folded into the exponents of pass 3
    float* loss;
    float* dlogits;
    int32_t* status;
    // Rows chosen by verification (accepted != null): row b of the launch is
    // position accepted[b] of sequence b when 0 <= accepted[b] < k (G = B, P = 1)
    // and its results go to slot r of a stable partition, active sequences first.
    const int32_t* accepted;
    int k;
    int32_t* seq_of_row;  // nullable: seq_of_row[r] = b
    int32_t* count;       // nullable: number of active sequences
    int csize;  // CTAs per row (cluster size)
    int span;   // vocabulary entries per CTA (multiple of 64)
};

// Pass-1 partial of a span: maxima, sums of 2^((x-m) log2 e) and one loss moment.
struct Stats1 {
    float mz, Ez, mt, Et, X;
    int err;
    int idx;   // CE: first index of the target maximum
    float zy;  // CE: draft logit at that index; RKL: the pivot target logit
};
// Pass-2 partial: JSD (KL(p||m), KL(q||m) in bits), or TVD (sum |p - q|,
// Q+ = sum of q over entries with q >= p, Q- = sum of q over q < p).
struct Stats2 {
    float a, b, c;
};

// RKL: the draft maximum with the target logit at it (the larger one on ties),
// merged in the same round as the target maximum.
__device__ __forceinline__ bool pivot_wins(float m, float t, float m0, float t0) {
    return m > m0 || (m == m0 && t > t0);
}
template <int kT>
__device__ __forceinline__ float3 block_max_pivot(float mz, float tp, float mt, float3* scratch) {
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, mz, o), t2 = __shfl_xor_sync(0xffffffffu, tp, o);
        if (pivot_wins(m2, t2, mz, tp)) { mz = m2; tp = t2; }
        mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, o));
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) scratch[warp] = make_float3(mz, tp, mt);
    __syncthreads();
    float3 r = scratch[0];
#pragma unroll
    for (int w = 1; w < kT / 32; ++w) {
        const float3 x = scratch[w];
        if (pivot_wins(x.x, x.y, r.x, r.y)) { r.x = x.x; r.y = x.y; }
        r.z = fmaxf(r.z, x.z);
    }
    return r;
}
// CE label: the target maximum with the lowest index, and the draft logit there.
struct Label {
    float m;
    int i;
    float z;
};
__device__ __forceinline__ Label merge_label(Label a, Label b) {
    return (b.m > a.m || (b.m == a.m && b.i < a.i)) ? b : a;
}

// Write one (exactly representable) value back to a staged row.
__device__ __forceinline__ void store_elem(float* p, float x) { *p = x; }
__device__ __forceinline__ void store_elem(__nv_bfloat16* p, float x) {
    *reinterpret_cast<unsigned short*>(p) = static_cast<unsigned short>(__float_as_uint(x) >> 16);
}

// TVD keeps q' = q sign(q - p) (fp32) in the two 16-bit (bf16) or the first
// 32-bit (fp32) staging slots of each entry once pass 2 has read its logits.
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}
template <typename In, int kCnt>
__device__ __forceinline__ void store_q(In* zs, In* ts, int j0, const float* q) {
    if constexpr (sizeof(In) == 4) {
        if constexpr (kCnt == 4) {
            *reinterpret_cast<float4*>(zs + j0) = make_float4(q[0], q[1], q[2], q[3]);
        } else {
#pragma unroll
            for (int e = 0; e < kCnt; ++e) reinterpret_cast<float*>(zs)[j0 + e] = q[e];
        }
    } else if constexpr (kCnt == 8) {
        uint32_t hz[4], ht[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t a = __float_as_uint(q[2 * i]), b = __float_as_uint(q[2 * i + 1]);
            hz[i] = prmt(a, b, 0x7632);  // high halves
            ht[i] = prmt(a, b, 0x5410);  // low halves
        }
        *reinterpret_cast<uint4*>(zs + j0) = make_uint4(hz[0], hz[1], hz[2], hz[3]);
        *reinterpret_cast<uint4*>(ts + j0) = make_uint4(ht[0], ht[1], ht[2], ht[3]);
    } else {
#pragma unroll
        for (int e = 0; e < kCnt; ++e) {
            const uint32_t a = __float_as_uint(q[e]);
            reinterpret_cast<unsigned short*>(zs)[j0 + e] = static_cast<unsigned short>(a >> 16);
            reinterpret_cast<unsigned short*>(ts)[j0 + e] = static_cast<unsigned short>(a & 0xffffu);
        }
    }
}
template <typename In>
__device__ __forceinline__ float load_q(const In* zs, const In* ts, int j) {
    if constexpr (sizeof(In) == 4) {
        return reinterpret_cast<const float*>(zs)[j];
    } else {
        const uint32_t hi = reinterpret_cast<const unsigned short*>(zs)[j];
        const uint32_t lo = reinterpret_cast<const unsigned short*>(ts)[j];
        return __uint_as_float((hi << 16) | lo);
    }
}
// With s = sign(q - p), G = sum_k q_k s_k / 2 and Q+ + Q- = sum q = 1, the TVD
// gradient q (s/2 - G) / tau is q Q- / tau where q >= p and -q Q+ / tau where
// q < p: both products of positive sums, so nothing cancels when one side
// holds almost all the mass.
template <typename In, bool kAligned, int kT>
__device__ __forceinline__ void tvd_gradient(const In* zs, const In* ts, int n, float gpos, float gneg,
                                             float* orow) {
    const int tid = threadIdx.x;
    auto g_of = [gpos, gneg](float q) { return q * (__float_as_int(q) < 0 ? gneg : gpos); };
    // the factor of q': gpos, or gneg where the sign bit is set (one shift and one
    // three-input logic op), so that the products go two at a time
    const uint32_t fpos = __float_as_uint(gpos), fdiff = fpos ^ __float_as_uint(gneg);
    auto factor = [fpos, fdiff](float q) {
        const uint32_t neg = static_cast<uint32_t>(__float_as_int(q) >> 31);
        return __uint_as_float(fpos ^ (neg & fdiff));
    };
    if constexpr (kAligned) {
        constexpr int kVec = Elem<In>::kVec;
        const int nv = n / kVec;
        for (int v = tid; v < nv; v += kT) {
            float q[kVec];
            if constexpr (sizeof(In) == 4) {
                const float4 f = *reinterpret_cast<const float4*>(zs + v * kVec);
                q[0] = f.x; q[1] = f.y; q[2] = f.z; q[3] = f.w;
            } else {
                const uint4 hz = lds_v4(zs + v * kVec), ht = lds_v4(ts + v * kVec);
                const uint32_t zw[4] = {hz.x, hz.y, hz.z, hz.w}, tw[4] = {ht.x, ht.y, ht.z, ht.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    q[2 * i] = __uint_as_float(prmt(tw[i], zw[i], 0x5410));
                    q[2 * i + 1] = __uint_as_float(prmt(tw[i], zw[i], 0x7632));
                }
            }
            float g[kVec];
#pragma unroll
            for (int e = 0; e < kVec; e += 2) {
                const float2 r = mul2(make_float2(q[e], q[e + 1]), make_float2(factor(q[e]), factor(q[e + 1])));
                g[e] = r.x;
                g[e + 1] = r.y;
            }
#pragma unroll
            for (int e = 0; e < kVec; e += 4) stg_v4(orow + v * kVec + e, g[e], g[e + 1], g[e + 2], g[e + 3]);
        }
        const int r0 = nv * kVec;
        if (tid < n - r0) orow[r0 + tid] = g_of(load_q(zs, ts, r0 + tid));
    } else {
        for (int e = tid; e < n; e += kT) orow[e] = g_of(load_q(zs, ts, e));
    }
}

template <typename In, int kKind, bool kAligned, int kT>
__global__ void __launch_bounds__(kT) distill_kernel(DistParams p) {
    // JSD clamps both rows to -1e30: a zero probability then stays exactly 0 and
    // every logit difference finite, so no entry needs a guard.  TVD needs none
    // either: a -inf gives p or q = 0, and the sign it picks multiplies q = 0.
    // FKL and RKL keep -inf (their loss is +inf when one row has mass where the
    // other has none) and guard only the 16-byte chunks that hold a -inf.
    constexpr bool kClamp = kKind == OSD_JSD;
    constexpr bool kClampZ = kClamp, kClampT = kClamp;
    constexpr bool kMoment = kKind == OSD_FKL || kKind == OSD_RKL;
    constexpr bool kNeedEt = kKind != OSD_CE;  // CE needs only the draft normaliser and the label
    constexpr bool kFold = !kClamp;            // exponent arguments by one FMA (see pass 1)
    // chunk loops unrolled by two where that measured faster: pass 0 of every kind (with
    // the scans below, RKL +2.3 %), passes 1-2 of TVD, JSD and CE (+2-3 %; FKL and RKL
    // lose 1-2 %), and JSD's gradient pass (the other kinds' lose 1-4 %)
    constexpr int kUn0 = 2;
    constexpr int kUn = (kKind == OSD_FKL || kKind == OSD_RKL) ? 1 : 2;
    constexpr int kUn3 = (kKind == OSD_JSD) ? 2 : 1;
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ Stats1 s1_mine, s1_all;
    __shared__ Stats2 s2_mine, s2_all;
    __shared__ float2 red_m[kT / 32];
    __shared__ float3 red_s[kT / 32];
    __shared__ int s_err;
    __shared__ float s_cu, s_cv, s_loss, s_K, s_tp;
    __shared__ Label red_l[kT / 32];
    __shared__ int2 red_i[kT / 32];

    const int tid = threadIdx.x;
    const int csize = p.csize;
    const float c = p.c, inv_tau = p.inv_tau;
    const int rank = (csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    long long row = blockIdx.x / csize;  // the launch row; from here on, the output row
    long long g, pp;
    const int V = p.V;
    const int e0 = rank * p.span;
    const int n = min(p.span, V - e0);
    In* zs = reinterpret_cast<In*>(dsm);
    In* ts = zs + p.span;
    bool issued = false;  // accepted mode: the span's copies went out before the slot count
    if (p.accepted) {
        // sequence b = row keeps position a = accepted[b] when a < k (the first rejected
        // draft token); the output slot counts the active sequences before it
        const int b = static_cast<int>(row), a = p.accepted[b];
        const bool active = a >= 0 && a < p.k;
        if (active) {  // the copies first: the count below runs while they are in flight
            stage_span_issue<In, kAligned>(zs, ts, static_cast<const In*>(p.draft) + b * p.dsg + a * p.dsp + e0,
                                           static_cast<const In*>(p.target) + b * p.tsg + a * p.tsp + e0, n,
                                           &bar, &s_err);
            issued = true;
        }
        int2 cnt = make_int2(0, 0);  // (active before b, active in total)
        for (int i = tid; i < p.G; i += kT) {
            const int ai = p.accepted[i];
            const int act = (ai >= 0 && ai < p.k) ? 1 : 0;
            cnt.x += (i < b) ? act : 0;
            cnt.y += act;
        }
        cnt = block_reduce<kT>(cnt, [](int2 u, int2 v) { return make_int2(u.x + v.x, u.y + v.y); },
                                         red_i);
        const long long slot = active ? cnt.x : cnt.y + (b - cnt.x);
        if (rank == 0 && tid == 0) {
            if (p.seq_of_row) p.seq_of_row[slot] = b;
            if (p.count && b == 0) *p.count = cnt.y;
        }
        row = slot;
        if (!active) {  // uniform over the cluster
            if (rank == 0 && tid == 0) p.loss[row] = 0.f;
            return;
        }
        g = b;
        pp = a;
    } else {
        if (p.mask && !p.mask[row]) {  // uniform over the cluster; no shared memory is exchanged
            if (rank == 0 && tid == 0) p.loss[row] = 0.f;
            return;
        }
        g = row / p.P;
        pp = row - g * p.P;
    }
    const In* zrow = static_cast<const In*>(p.draft) + g * p.dsg + pp * p.dsp;
    const In* trow = static_cast<const In*>(p.target) + g * p.tsg + pp * p.tsp;

    // ---- stage the span of both rows in shared memory
    const int err_local = issued ? stage_span_land<In, kAligned, kT>(zs, ts, zrow + e0, trow + e0, n, &bar, &s_err)
                                 : stage_span<In, kAligned, kT>(zs, ts, zrow + e0, trow + e0, n, &bar, &s_err);

    // ---- pass 0: this thread's maxima, and the chunk where each first appears
    float mz = kNegInf, mt = kNegInf;
    int jz = -1, jt = -1;
    if (!err_local) {
        sweep<In, kAligned, kClampZ, kClampT, true, false, kUn0, kT>(zs, ts, n, [&](const float* z, const float* t, auto tag,
                                                                   int j0, float cz, float ct, bool,
                                                                   const uint4& zr, const uint4& tr) {
            if (cz > mz) { mz = cz; jz = j0; }
            if (ct > mt) { mt = ct; jt = j0; }
            if constexpr (kClamp) {  // clamp the staged logits once, for every later pass
                if constexpr (decltype(tag)::value > 1) {
                    *reinterpret_cast<uint4*>(zs + j0) = zr;
                    *reinterpret_cast<uint4*>(ts + j0) = tr;
                } else {
                    store_elem(zs + j0, z[0]);
                    store_elem(ts + j0, t[0]);
                }
            }
        });
    }
    // the entry that holds a maximum: RKL's pivot target logit, CE's label
    auto chunk_len = [n](int j0) {
        constexpr int kVec = Elem<In>::kVec;
        return (kAligned && j0 < (n / kVec) * kVec) ? kVec : 1;
    };
    float tp = 0.f;                      // RKL: target logit at this thread's draft maximum
    Label lab{kNegInf, INT_MAX, 0.f};    // CE: this thread's first target maximum
    // (the scans are unrolled over a whole chunk, predicated on its length, so that
    // their shared-memory loads go out together: RKL +1.5 %)
    if (kKind == OSD_RKL && jz >= 0) {
        const int cnt = chunk_len(jz);
#pragma unroll
        for (int e = Elem<In>::kVec - 1; e >= 0; --e)
            if (e < cnt && Elem<In>::lds(zs + jz + e) == mz) tp = Elem<In>::lds(ts + jz + e);
        if (tp == kNegInf) tp = 0.f;  // any finite pivot works; the loss is +inf then anyway
    }
    if (kKind == OSD_CE && jt >= 0) {
        const int cnt = chunk_len(jt);
        int ei = 0;
#pragma unroll
        for (int e = Elem<In>::kVec - 1; e >= 0; --e)
            if (e < cnt && Elem<In>::lds(ts + jt + e) == mt) ei = e;
        lab = Label{mt, e0 + jt + ei, Elem<In>::lds(zs + jt + ei)};
    }
    // block maxima: every thread's sums of pass 1 then share one reference
    float gzb, gtb, tpv = 0.f;
    Label bl{kNegInf, INT_MAX, 0.f};
    if constexpr (kKind == OSD_RKL) {
        const float3 r = block_max_pivot<kT>(mz, tp, mt, red_s);
        gzb = r.x;
        tpv = r.y;
        gtb = r.z;
    } else {
        // red_m has no readers yet: staging ended on a block barrier
        const float2 bm = block_max2<false, kT>(mz, mt, red_m);
        gzb = bm.x;
        gtb = bm.y;
        if constexpr (kKind == OSD_CE)
            bl = block_reduce<kT>(lab, [](Label a, Label b) { return merge_label(a, b); }, red_l);
    }

    // ---- pass 1: sums of 2^((x - m) c) against the block maxima (+ the FKL/RKL moment)
    // The RKL moment is taken about a pivot, the draft maximum m_z and the target
    // logit t_pv found there: X = sum_j e_j ((z_j - m_z) - (t_j - t_pv)).  The
    // pivot's own term is exactly 0, so when q is nearly one-hot the gradient
    // q_j (log q_j - log p_j - loss) at the peak comes out as a sum of small
    // terms instead of the difference of two large ones.
    bool row_ninf = false;  // this thread saw a -inf logit (FKL, RKL)
    bool rkl_inf = false;   // RKL: a finite draft logit meets a -inf target logit
    float2 Ez2 = f2(0.f), Et2 = f2(0.f), X2 = f2(0.f);
    const bool zok = kClampZ || gzb != kNegInf;
    const bool tok = kNeedEt && (kClampT || gtb != kNegInf);
    // Exponent arguments.  Unclamped kinds take (x - m) c as one FMA, x c - M with
    // M = rn(m c): the rounding of M is a factor common to the whole row, so it
    // cancels in the normalisation, and the row constants below add back its
    // exact value fma(m, c, -M).  JSD keeps the exact difference, because its
    // -1e30 clamp would make x c - M cancel catastrophically on an all-clamped span.
    // A span with no mass gets M = 0: its logits are all -inf and so are x c - M.
    const float Mz = zok ? __fmul_rn(gzb, c) : 0.f, Mt = tok ? __fmul_rn(gtb, c) : 0.f;
    if (!err_local) {
        const float2 gz2 = f2(gzb), gt2 = f2(gtb), tp2 = f2(tpv);
        const float2 nMz2 = f2(-Mz), nMt2 = f2(-Mt);
        sweep<In, kAligned, false, false, false, kMoment, kUn, kT>(zs, ts, n, [&](const float* z, const float* t,
                                                                             auto tag, int, float, float,
                                                                             bool ninf, const uint4&, const uint4&) {
            constexpr int kCnt = decltype(tag)::value;
            row_ninf |= ninf;
            if (kCnt == 1 || ninf) {  // element-wise, with the guards a -inf needs
#pragma unroll
                for (int e = 0; e < kCnt; ++e) {
                    if (zok) {
                        const float ez = kFold ? ex2(fmaf(z[e], c, -Mz)) : ex2((z[e] - gzb) * c);
                        Ez2.x += ez;
                        if (kKind == OSD_RKL && z[e] != kNegInf) {
                            if (t[e] == kNegInf) rkl_inf = true;  // q > 0 = p: the loss is +inf
                            else X2.x = fmaf(ez, (z[e] - gzb) - (t[e] - tpv), X2.x);
                        }
                    }
                    if (tok) {
                        const float et = kFold ? ex2(fmaf(t[e], c, -Mt)) : ex2((t[e] - gtb) * c);
                        Et2.x += et;
                        if (kKind == OSD_FKL && et > 0.f) X2.x = fmaf(et, t[e] - z[e], X2.x);
                    }
                }
            } else {
                // no -inf in the chunk, and (unclamped) every span with finite logits has
                // zok / tok set, so the sums need no per-chunk condition
#pragma unroll
                for (int e = 0; e < kCnt; e += 2) {
                    const float2 zz = make_float2(z[e], z[e + 1]);
                    float2 a;
                    if constexpr (kFold) a = fma2(zz, f2(c), nMz2);
                    else a = mul2(sub2(zz, gz2), f2(c));
                    const float2 ez = make_float2(ex2(a.x), ex2(a.y));
                    Ez2 = add2(Ez2, ez);
                    if (kKind == OSD_RKL)
                        X2 = fma2(ez, sub2(sub2(zz, gz2), sub2(make_float2(t[e], t[e + 1]), tp2)), X2);
                }
                if constexpr (kNeedEt) {
#pragma unroll
                    for (int e = 0; e < kCnt; e += 2) {
                        const float2 tt = make_float2(t[e], t[e + 1]);
                        float2 a;
                        if constexpr (kFold) a = fma2(tt, f2(c), nMt2);
                        else a = mul2(sub2(tt, gt2), f2(c));
                        const float2 et = make_float2(ex2(a.x), ex2(a.y));
                        Et2 = add2(Et2, et);
                        if (kKind == OSD_FKL) X2 = fma2(et, sub2(tt, make_float2(z[e], z[e + 1])), X2);
                    }
                }
            }
        });
    }
    {
        // red_s was last read by RKL's pivot merge; the other kinds have not used it yet
        const float3 bs = block_sum3<kKind == OSD_RKL, kT>(Ez2.x + Ez2.y, Et2.x + Et2.y, X2.x + X2.y, red_s);
        const int any_ninf = kMoment ? __syncthreads_or(row_ninf ? 1 : 0) : 0;
        const int any_inf = (kKind == OSD_RKL) ? __syncthreads_or(rkl_inf ? 1 : 0) : 0;
        if (tid == 0)
            s1_mine = Stats1{gzb, bs.x, (kKind == OSD_CE) ? bl.m : gtb, bs.y, bs.z,
                             err_local | (any_ninf << 1) | (any_inf << 2), bl.i,
                             (kKind == OSD_RKL) ? tpv : bl.z};
    }
    // cluster merge: warp 0 gathers every CTA's partial (lane r <- CTA r) and reduces
    // it in a fixed order, so all CTAs of the row hold bit-identical statistics
    if (csize > 1) cluster_sync_publish(tid == 0); else __syncthreads();
    if (tid < 32) {
        Stats1 o{kNegInf, 0.f, kNegInf, 0.f, 0.f, 0, INT_MAX, 0.f};
        if (tid < csize) {
            if (tid == rank) {
                o = s1_mine;
            } else {
                const uint32_t base = map_rank(&s1_mine, tid);
                o.mz = ld_dsmem_f32(base + offsetof(Stats1, mz));
                o.Ez = ld_dsmem_f32(base + offsetof(Stats1, Ez));
                o.mt = ld_dsmem_f32(base + offsetof(Stats1, mt));
                o.Et = ld_dsmem_f32(base + offsetof(Stats1, Et));
                o.X = ld_dsmem_f32(base + offsetof(Stats1, X));
                o.err = ld_dsmem_s32(base + offsetof(Stats1, err));
                if (kKind == OSD_CE) o.idx = ld_dsmem_s32(base + offsetof(Stats1, idx));
                if (kKind == OSD_CE || kKind == OSD_RKL) o.zy = ld_dsmem_f32(base + offsetof(Stats1, zy));
            }
        }
        Label L{o.mt, o.idx, o.zy};  // CE label: the CTA labels merge like an argmax
        if constexpr (kKind == OSD_CE) {
            for (int off = 16; off > 0; off >>= 1) {
                const Label w{__shfl_xor_sync(0xffffffffu, L.m, off), __shfl_xor_sync(0xffffffffu, L.i, off),
                              __shfl_xor_sync(0xffffffffu, L.z, off)};
                L = merge_label(L, w);
            }
        }
        float gz = o.mz, gt = o.mt;
        int err = o.err;
        for (int off = 16; off > 0; off >>= 1) {
            gz = fmaxf(gz, __shfl_xor_sync(0xffffffffu, gz, off));
            gt = fmaxf(gt, __shfl_xor_sync(0xffffffffu, gt, off));
            err |= __shfl_xor_sync(0xffffffffu, err, off);
        }
        // each CTA's sums are against 2^(M_cta) (folded kinds) or 2^(m_cta c): bring them to the row's
        auto to_row = [c](float m, float g) {
            if (m == kNegInf) return 0.f;
            return kFold ? ex2(__fmul_rn(m, c) - __fmul_rn(g, c)) : ex2((m - g) * c);
        };
        const float sz = to_row(o.mz, gz), st = to_row(o.mt, gt);
        float tg = 0.f;  // RKL: the row's pivot target logit
        if constexpr (kKind == OSD_RKL) {
            tg = (o.mz == gz && o.mz != kNegInf) ? o.zy : kNegInf;
            for (int off = 16; off > 0; off >>= 1) tg = fmaxf(tg, __shfl_xor_sync(0xffffffffu, tg, off));
            if (tg == kNegInf) tg = 0.f;
        }
        float Ez = o.Ez * sz, Et = o.Et * st, X;
        if constexpr (kKind == OSD_RKL)
            X = (o.mz == kNegInf) ? 0.f : fmaf(o.Ez, (o.mz - gz) - (o.zy - tg), o.X) * sz;
        else
            X = o.X * st;
        for (int off = 16; off > 0; off >>= 1) {
            Ez += __shfl_xor_sync(0xffffffffu, Ez, off);
            Et += __shfl_xor_sync(0xffffffffu, Et, off);
            X += __shfl_xor_sync(0xffffffffu, X, off);
        }
        if (tid == 0) {
            s1_all = Stats1{gz, Ez, gt, Et, X, err, L.i, L.z};
            // row constants, computed once: log2 p = (t - m_t) c - log2(E_t) with
            // c = log2(e)/tau; the difference is exact, so the rounding never scales
            // with the size of the logits.  Folded sums are against 2^M, M = rn(m c):
            // E' = E 2^dm with dm = m c - M, taken exactly by an FMA
            float dz = 0.f, dt = 0.f;
            if (kFold) {
                if (gz != kNegInf) dz = fmaf(gz, c, -__fmul_rn(gz, c));
                if (gt != kNegInf) dt = fmaf(gt, c, -__fmul_rn(gt, c));
            }
            s_cu = -log2f(Et) + dt;
            s_cv = -log2f(Ez) + dz;
            const float lr = logf(Ez / Et) - kLn2 * (dz - dt);
            float l = 0.f;
            if (kKind == OSD_FKL) l = (X / Et - (gt - gz)) * inv_tau + lr;
            // RKL about the pivot: loss = log q - log p at the pivot + sum_j q_j D_j, with
            // D_j = ((z_j - m_z) - (t_j - t_pv)) / tau; s_K keeps the sum for pass 3
            if (kKind == OSD_RKL) l = (err & 4) ? __builtin_huge_valf() : (X / Ez + (gt - tg)) * inv_tau - lr;
            if (kKind == OSD_CE) l = (gz - L.z) * inv_tau + (logf(Ez) - kLn2 * dz);  // -log q(y*)
            s_loss = l;
            s_K = X / Ez * inv_tau;
            s_tp = tg;
        }
    }
    __syncthreads();
    const Stats1 st = s1_all;
    const bool row_err = (st.err & 1) != 0;
    const bool has_ninf = (st.err & 2) != 0;  // some logit of the row is -inf
    const float cu = s_cu, cv = s_cv;
    const float2 mt2 = f2(st.mt), mz2 = f2(st.mz);
    auto log2p = [&](float2 x) { return fma2(sub2(x, mt2), f2(c), f2(cu)); };  // pass 2
    auto log2q = [&](float2 x) { return fma2(sub2(x, mz2), f2(c), f2(cv)); };
    float loss = s_loss;

    const float beta = p.beta;
    const bool jsd_trivial = (kKind == OSD_JSD) && (beta == 0.f || beta == 1.f);  // m = q or m = p: loss 0
    Stats2 s2 = {0.f, 0.f, 0.f};
    if constexpr (kKind == OSD_JSD || kKind == OSD_TVD) {
        // ---- pass 2: divergence terms with the global normalisers
        float2 A2 = f2(0.f), B2 = f2(0.f), C2 = f2(0.f);
        if (!row_err && !jsd_trivial) {
            sweep<In, kAligned, false, false, false, false, kUn, kT>(zs, ts, n, [&](const float* z, const float* t,
                                                                               auto tag, int j0, float, float, bool,
                                                                               const uint4& zr, const uint4& tr) {
                constexpr int kCnt = decltype(tag)::value;
                // TVD's bf16 chunks: x - m straight from the packed words the sweep loaded
                // (measured, JSD does as well unpacking)
                constexpr bool kRaw = sizeof(In) == 2 && kCnt == 8 && kKind == OSD_TVD;
                const uint32_t zw[4] = {zr.x, zr.y, zr.z, zr.w}, tw[4] = {tr.x, tr.y, tr.z, tr.w};
                float qs[kCnt];  // TVD: q sign(q - p), kept for pass 3
#pragma unroll
                for (int e = 0; e < kCnt; e += 2) {
                    const bool two = (e + 1 < kCnt);
                    float2 u, v;  // log2 p, log2 q
                    if constexpr (kRaw) {
                        u = fma2(bf16x2_minus(tw[e / 2], st.mt), f2(c), f2(cu));
                        v = fma2(bf16x2_minus(zw[e / 2], st.mz), f2(c), f2(cv));
                    } else {
                        u = log2p(make_float2(t[e], two ? t[e + 1] : t[e]));
                        v = log2q(make_float2(z[e], two ? z[e + 1] : z[e]));
                    }
                    float2 a, b, c2 = f2(0.f);
                    if (kKind == OSD_TVD) {
                        const float2 pj = make_float2(ex2(u.x), ex2(u.y)), qj = make_float2(ex2(v.x), ex2(v.y));
                        const float2 df = sub2(qj, pj);
                        a = make_float2(fabsf(df.x), fabsf(df.y));
                        const float2 qq = make_float2(copysignf(qj.x, df.x), copysignf(qj.y, df.y));  // q sign(q - p)
                        qs[e] = qq.x;
                        if (e + 1 < kCnt) qs[e + 1] = qq.y;
                        b = add2(qj, qq);   // 2q where q >= p, else 0 (exact): into 2 Q+
                        c2 = sub2(qj, qq);  // 2q where q < p, else 0: into 2 Q-
                    } else {
                        // p log2(p/m), q log2(q/m): log2 p, log2 q exact from the logits, log2 m
                        // by one lg2 (m floored at the smallest normal, where lg2 would flush;
                        // the entry's p and q are negligible there)
                        const float2 pj = make_float2(ex2(u.x), ex2(u.y)), qj = make_float2(ex2(v.x), ex2(v.y));
                        const float2 m = fma2(pj, f2(beta), mul2(qj, f2(1.f - beta)));
                        const float2 lm = make_float2(lg2(fmaxf(m.x, kMinNormal)), lg2(fmaxf(m.y, kMinNormal)));
                        // straight into the sums (the second slot of a one-entry chunk
                        // carries no mass); JSD has no third sum
                        const float2 pw = two ? pj : make_float2(pj.x, 0.f);
                        const float2 qw = two ? qj : make_float2(qj.x, 0.f);
                        A2 = fma2(pw, sub2(u, lm), A2);
                        B2 = fma2(qw, sub2(v, lm), B2);
                        continue;
                    }
                    if (!two) { a.y = 0.f; b.y = 0.f; c2.y = 0.f; }
                    A2 = add2(A2, a);
                    B2 = add2(B2, b);
                    C2 = add2(C2, c2);
                }
                // the logits of these entries are not needed again: their slots take q'
                if constexpr (kKind == OSD_TVD) store_q<In, kCnt>(zs, ts, j0, qs);
            });
        }
        // red_s was last read before the cluster merge's barriers
        const float3 bs = block_sum3<false, kT>(A2.x + A2.y, B2.x + B2.y, C2.x + C2.y, red_s);
        if (tid == 0) s2_mine = Stats2{bs.x, bs.y, bs.z};
        if (csize > 1) cluster_sync_publish(tid == 0); else __syncthreads();
        if (tid < 32) {
            float a = 0.f, b = 0.f, cc = 0.f;
            if (tid < csize) {
                if (tid == rank) {
                    a = s2_mine.a;
                    b = s2_mine.b;
                    cc = s2_mine.c;
                } else {
                    const uint32_t base = map_rank(&s2_mine, tid);
                    a = ld_dsmem_f32(base + offsetof(Stats2, a));
                    b = ld_dsmem_f32(base + offsetof(Stats2, b));
                    if (kKind == OSD_TVD) cc = ld_dsmem_f32(base + offsetof(Stats2, c));
                }
            }
            for (int off = 16; off > 0; off >>= 1) {
                a += __shfl_xor_sync(0xffffffffu, a, off);
                b += __shfl_xor_sync(0xffffffffu, b, off);
                if (kKind == OSD_TVD) cc += __shfl_xor_sync(0xffffffffu, cc, off);
            }
            if (tid == 0) s2_all = Stats2{a, b, cc};
        }
        __syncthreads();
        s2 = s2_all;
        if (kKind == OSD_TVD) {
            loss = 0.5f * s2.a;
            s2.b *= 0.5f;
            s2.c *= 0.5f;
        } else {
            loss = jsd_trivial ? 0.f : kLn2 * (beta * s2.a + (1.f - beta) * s2.b);
        }
    }
    if (csize > 1) cluster_arrive_relaxed();  // finished reading the other CTAs' shared memory

    if (rank == 0 && tid == 0) {
        p.loss[row] = row_err ? __int_as_float(0x7fc00000) : loss;
        if (row_err && p.status) atomicExch(p.status, static_cast<int32_t>(OSD_ERR_TIMEOUT));
    }

    // ---- pass 3: d loss / d draft logits of the span
    if (kKind == OSD_TVD && !row_err) {
        // from the stored q' = q sign(q - p): q' Q- / tau, or q' Q+ / tau where q' < 0
        tvd_gradient<In, kAligned, kT>(zs, ts, n, s2.c * inv_tau, s2.b * inv_tau, p.dlogits + row * V + e0);
    } else if (kKind != OSD_TVD && !row_err) {
        float* orow = p.dlogits + row * V + e0;
        const float K = s_K, tpg = s_tp;
        // q and p of this pass come out multiplied by the gradient's constant factor
        const float2 cvs = f2(cv + p.lg_scale), cus = f2(cu + p.lg_scale);
        const int label = st.idx;
        bool own_label = false;  // CE: this thread's stores hold the label's entry
        sweep<In, kAligned, false, false, false, false, kUn3, kT>(zs, ts, n, [&](const float* z, const float* t,
                                                                            auto tag, int j0, float, float, bool,
                                                                            const uint4& zr, const uint4& tr) {
            constexpr int kCnt = decltype(tag)::value;
            // bf16 chunks of FKL/RKL, which need x - m of both rows, take the differences straight
            // from the packed words (mixed-precision subtracts) instead of unpacking first;
            // measured, CE and JSD do better unpacking
            constexpr bool kRaw = sizeof(In) == 2 && kCnt == 8 && (kKind == OSD_FKL || kKind == OSD_RKL);
            const uint32_t zw[4] = {zr.x, zr.y, zr.z, zr.w}, tw[4] = {tr.x, tr.y, tr.z, tr.w};
            // x - m of the pair at e, from the packed words or the unpacked values
            auto zdiff = [&](int e, float m) {
                if constexpr (kRaw) return bf16x2_minus(zw[e / 2], m);
                else return sub2(make_float2(z[e], (e + 1 < kCnt) ? z[e + 1] : z[e]), f2(m));
            };
            auto tdiff = [&](int e, float m) {
                if constexpr (kRaw) return bf16x2_minus(tw[e / 2], m);
                else return sub2(make_float2(t[e], (e + 1 < kCnt) ? t[e + 1] : t[e]), f2(m));
            };
            float gr[kCnt];
#pragma unroll
            for (int e = 0; e < kCnt; e += 2) {
                const bool two = (e + 1 < kCnt);
                const float2 zd = zdiff(e, st.mz);
                const float2 v = fma2(zd, f2(c), cvs);  // log2 q + lg_scale
                const float2 qj = make_float2(ex2(v.x), ex2(v.y));
                float2 gg;
                if (kKind == OSD_FKL) {  // (q - p) / tau
                    const float2 u = fma2(tdiff(e, st.mt), f2(c), cus);
                    gg = sub2(qj, make_float2(ex2(u.x), ex2(u.y)));
                } else if (kKind == OSD_CE) {  // (q - onehot(y*)) / tau
                    const int j = e0 + j0 + e;
                    const bool lx = (j == label), ly = (j + 1 == label);
                    own_label |= lx || (two && ly);
                    gg = sub2(qj, make_float2(lx ? inv_tau : 0.f, ly ? inv_tau : 0.f));
                } else if (kKind == OSD_RKL) {  // q_j (D_j - sum_k q_k D_k) / tau
                    const float2 dd = sub2(zd, tdiff(e, tpg));
                    gg = mul2(qj, fma2(dd, f2(inv_tau), f2(-K)));
                    if (has_ninf) {  // q = 0 against an infinite log-ratio contributes 0
                        if (!(qj.x > 0.f)) gg.x = 0.f;
                        if (!(qj.y > 0.f)) gg.y = 0.f;
                    }
                } else {
                    if (jsd_trivial) {
                        gg = f2(0.f);
                    } else {
                        // q (log2(q/m) - S), every probability here carrying the gradient's
                        // factor, which cancels in log2(q/m)
                        const float2 u = fma2(tdiff(e, st.mt), f2(c), cus);
                        const float2 pj = make_float2(ex2(u.x), ex2(u.y));
                        const float2 m = fma2(pj, f2(beta), mul2(qj, f2(1.f - beta)));
                        const float2 lm = make_float2(lg2(fmaxf(m.x, kMinNormal)), lg2(fmaxf(m.y, kMinNormal)));
                        gg = mul2(qj, sub2(sub2(v, lm), f2(s2.b)));
                    }
                }
                gr[e] = gg.x;
                if (two) gr[e + 1] = gg.y;
            }
            if constexpr (kAligned && kCnt >= 4) {
#pragma unroll
                for (int e = 0; e < kCnt; e += 4) stg_v4(orow + j0 + e, gr[e], gr[e + 1], gr[e + 2], gr[e + 3]);
            } else {
#pragma unroll
                for (int e = 0; e < kCnt; ++e) orow[j0 + e] = gr[e];
            }
        });
        // CE: at the label q / tau - 1 / tau keeps only the resolution of 1 / tau (an ulp
        // of 1.43 at tau = 0.7, where q is near 1); the thread that stored the entry writes
        // it again as (q - 1) / tau, with q - 1 exact (a CTA barrier before a write by one
        // fixed thread cost CE 6 %)
        if (kKind == OSD_CE && own_label) orow[label - e0] = (ex2(fmaf(st.zy - st.mz, c, cv)) - 1.f) * inv_tau;
    }
    if (csize > 1) cluster_wait();  // keep this CTA's statistics readable until every peer is done
}

// ------------------------------------------------------------------ TMEM-staged runs of rows
// The same passes over the same spans, but each cluster walks a run of up to
// kTmRows consecutive rows (the last runs shorter, see launch_distill_tm).  A row's span lands in shared memory by bulk copy
// as above, is moved at once into tensor memory (each thread owns one
// tensor-memory lane and keeps its 16-byte chunks in that lane's columns), and
// the next active row's bulk copy then goes into the freed shared memory while
// this row's passes read tensor memory: the copy of row i+1 overlaps the passes
// of row i, with the shared-memory footprint of one staged span per CTA.  The
// hardware schedules the runs like any grid (no assumption on how many
// clusters are resident), and masked-out rows of a run cost one mask read.
// 16-byte-aligned rows; TVD, JSD, RKL and FKL (CE, which needs no second
// exchange, stays on the per-row kernel, at 97 % of the HBM peak there).  A row
// costs one CTA barrier (the staging buffer is free) and two exchanges within
// the cluster: TVD and JSD exchange the normalisers, then the sums of pass 2;
// RKL and FKL the maxima (RKL with its pivot), then the sums and the moment.
constexpr int kTmThreads = 128;  // one warp per tensor-memory lane quarter
constexpr int kTmG = 2;          // chunk slots per round of tensor-memory loads
constexpr int kTmRows = 8;       // rows per cluster run
constexpr int kTmJsdG = 1;       // JSD's passes 2 and 3: one chunk slot per round (no spills at 72 registers)
constexpr int kTmMomG = 1;       // RKL and FKL pass 1: one chunk slot per round (no spills at 72 registers)
constexpr int kTmMaxChunks = 4096;  // 16-byte chunks per span (<= 256 columns; longer spans stage as above)

struct TmShape {
    int slots;       // 16-byte chunks of each row per thread
    int t_off;       // first column of the target words (z words from column 0)
    uint32_t ncols;  // tensor-memory columns per CTA
    // runs, longest first: rows [0, end8) in runs of `run` (8, 4 or 2; twice that
    // under a mask), [end8, end2) in runs of piece2, then runs of piece1 rows; n8 and
    // n2 runs of the first two kinds
    long long end8, end2;
    int n8, n2;
    int run;
    int piece2, piece1;  // rows of the two kinds of tail pieces (2 and 1; 6 and 3 under a mask)
};

// This thread's chunks of a span held in tensor memory: slot s is chunk
// v = tid + kTmThreads s (entries v kVec ..), its draft words in columns
// 4s .. 4s+3 and its target words in t_off + 4s ..; then the ragged tail of
// fewer than kVec entries, one per thread tid < tail, kept in that thread's
// registers (tz, tt).  f is `sweep`'s callback, with the chunk's packed words by
// reference: kStore writes them back.
template <typename In, bool kClampZ, bool kClampT, bool kMax, bool kMin, bool kStore, int kG = kTmG, typename F>
__device__ __forceinline__ void sweep_tm(uint32_t tw, const TmShape& sh, int nv, int tail, float& tz, float& tt,
                                         F&& f) {
    static_assert(kG == 1 || kG == kTmG, "one or kTmG chunk slots per round");
    using E = Elem<In>;
    constexpr int kVec = E::kVec;
    const int tid = threadIdx.x;
    for (int s0 = 0; s0 < sh.slots; s0 += kG) {
        uint4 zr[kG], tr[kG];
        if constexpr (kG == 1) {
            tm_ld4(tw + 4 * s0, zr[0]);
            tm_ld4(tw + sh.t_off + 4 * s0, tr[0]);
        } else {
            tm_ld8(tw + 4 * s0, zr[0], zr[1]);
            tm_ld8(tw + sh.t_off + 4 * s0, tr[0], tr[1]);
        }
        tm_wait_ld();
#pragma unroll
        for (int g = 0; g < kG; ++g) {
            const int v = tid + kTmThreads * (s0 + g);
            if (v < nv) {
                if (kClampZ) E::clamp_raw(zr[g]);
                if (kClampT) E::clamp_raw(tr[g]);
                float z[kVec], t[kVec];
                E::unpack(zr[g], z);
                E::unpack(tr[g], t);
                const float cz = kMax ? E::max_raw(zr[g]) : 0.f, ct = kMax ? E::max_raw(tr[g]) : 0.f;
                const bool ninf = kMin ? (fminf(E::min_raw(zr[g]), E::min_raw(tr[g])) == kNegInf) : false;
                f(z, t, std::integral_constant<int, kVec>{}, v * kVec, cz, ct, ninf, zr[g], tr[g]);
            }
        }
        if constexpr (kStore && kG == 1) {
            tm_st4(tw + 4 * s0, zr[0]);
            tm_st4(tw + sh.t_off + 4 * s0, tr[0]);
        } else if constexpr (kStore) {
            tm_st8(tw + 4 * s0, zr[0], zr[1]);
            tm_st8(tw + sh.t_off + 4 * s0, tr[0], tr[1]);
        }
    }
    if constexpr (kStore) tm_wait_st();
    if (tid < tail) {
        float z = tz, t = tt;
        if (kClampZ) z = E::clamp1(z);
        if (kClampT) t = E::clamp1(t);
        uint4 dz{}, dt{};
        f(&z, &t, std::integral_constant<int, 1>{}, nv * kVec + tid, z, t, fminf(z, t) == kNegInf, dz, dt);
        if constexpr (kStore) { tz = z; tt = t; }
    }
}

// q' = q sign(q - p) of a chunk, packed into the chunk's words the way store_q
// packs it into the staging slots (bf16: high halves in the draft words, low
// halves in the target words; fp32: the draft words).
template <typename In>
__device__ __forceinline__ void pack_q(const float* q, uint4& zr, uint4& tr) {
    if constexpr (sizeof(In) == 4) {
        zr = make_uint4(__float_as_uint(q[0]), __float_as_uint(q[1]), __float_as_uint(q[2]), __float_as_uint(q[3]));
    } else {
        uint32_t hz[4], ht[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t a = __float_as_uint(q[2 * i]), b = __float_as_uint(q[2 * i + 1]);
            hz[i] = prmt(a, b, 0x7632);
            ht[i] = prmt(a, b, 0x5410);
        }
        zr = make_uint4(hz[0], hz[1], hz[2], hz[3]);
        tr = make_uint4(ht[0], ht[1], ht[2], ht[3]);
    }
}
template <typename In>
__device__ __forceinline__ void unpack_q(const uint4& zr, const uint4& tr, float* q) {
    if constexpr (sizeof(In) == 4) {
        q[0] = __uint_as_float(zr.x); q[1] = __uint_as_float(zr.y);
        q[2] = __uint_as_float(zr.z); q[3] = __uint_as_float(zr.w);
    } else {
        const uint32_t zw[4] = {zr.x, zr.y, zr.z, zr.w}, tw[4] = {tr.x, tr.y, tr.z, tr.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            q[2 * i] = __uint_as_float(prmt(tw[i], zw[i], 0x5410));
            q[2 * i + 1] = __uint_as_float(prmt(tw[i], zw[i], 0x7632));
        }
    }
}

// A row's statistics travel without cluster barriers.  In an exchange each warp
// leaves its value (the same in all its lanes) in a slot of its CTA and arrives
// on named barrier 1, where warp 0 waits; warp 0 merges the slots into the CTA's
// partial and pushes it with st.async into slot `rank` of every CTA's receive
// buffer for that exchange, completing 16 bytes on that CTA's barrier; it then
// merges the csize partials, in rank order, writes the result for the other
// warps and arrives on named barrier 2, where they wait.  Every CTA merges the
// same partials in the same order, so all reach the same bits.  A row makes two
// exchanges, each with its own receive buffer and barrier: a CTA pushes its
// next partial of an exchange only after every CTA's partial of the other one
// has reached it, which each peer sends only once it has read the buffer.
__device__ __forceinline__ float warp_max(float x) {
    for (int off = 16; off > 0; off >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, off));
    return x;
}
__device__ __forceinline__ float warp_sum(float x) {
    // the butterfly leaves the same bits in every lane (each step adds the same two values)
    for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
    return x;
}
__device__ __forceinline__ int warp_or(int x) {
    for (int off = 16; off > 0; off >>= 1) x |= __shfl_xor_sync(0xffffffffu, x, off);
    return x;
}
// RKL: the draft maximum with the target logit at it (the larger one on ties) in
// .x/.y of every lane
__device__ __forceinline__ float2 warp_max_pivot(float m, float t) {
    for (int off = 16; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, off), t2 = __shfl_xor_sync(0xffffffffu, t, off);
        if (pivot_wins(m2, t2, m, t)) {
            m = m2;
            t = t2;
        }
    }
    return make_float2(m, t);
}
// log2 of a sum of exponentials that is at least 1 (the term of the maximum):
// the exponent plus lg2.approx of the mantissa in [1, 2), absolute error about
// 2^-22 there; anything else (0 of a row with no mass, inf, NaN) straight through lg2.approx
__device__ __forceinline__ float log2_sum(float x) {
    if (!(x >= 1.f && x <= 3.0e38f)) return lg2(x);
    const uint32_t b = __float_as_uint(x);
    return static_cast<float>(static_cast<int>(b >> 23) - 127) + lg2(__uint_as_float((b & 0x007fffffu) | 0x3f800000u));
}
constexpr uint64_t kTmPartWaitNs = 3000000000ull;  // partials: peers may first wait out their copies
// Named barriers 1 and 2 of the CTA (0 is __syncthreads): `arrive` marks the
// warp's arrival without waiting (release), `sync` waits for all kTmThreads (acquire).
__device__ __forceinline__ void named_arrive(int id) {
    asm volatile("bar.arrive %0, %1;" :: "r"(id), "n"(kTmThreads) : "memory");
}
__device__ __forceinline__ void named_sync(int id) {
    asm volatile("bar.sync %0, %1;" :: "r"(id), "n"(kTmThreads) : "memory");
}
// The flags of an RKL row, OR-ed over the cluster in the .w of its second exchange.
constexpr int kTmNinf = 1;    // some logit is -inf
constexpr int kTmRklInf = 2;  // a finite draft logit meets a -inf target logit: the loss is +inf

template <typename In, int kKind>
__global__ void __launch_bounds__(kTmThreads, 7) distill_tm_kernel(DistParams p, TmShape tsh) {
    static_assert(kKind == OSD_TVD || kKind == OSD_JSD || kKind == OSD_RKL || kKind == OSD_FKL,
                  "the TMEM-staged runs serve TVD, JSD, RKL and FKL");
    constexpr int kT = kTmThreads, kW = kT / 32;
    constexpr int kVec = Elem<In>::kVec;
    constexpr bool kJsd = kKind == OSD_JSD, kTvd = kKind == OSD_TVD, kRkl = kKind == OSD_RKL;
    constexpr bool kFkl = kKind == OSD_FKL;
    constexpr bool kMom = kRkl || kFkl;  // the maxima go round first, then the sums with the loss moment
    // work done while the span moves into tensor memory: FKL's pass 0 (the maxima; 1.6 %
    // faster than a sweep of its own), JSD's clamp and its first-chunk maxima (below).
    // RKL keeps pass 0 as a sweep after the next row's copy is issued (1.9 % faster that way)
    constexpr bool kStage0 = kJsd || kFkl;
    // TVD and JSD need no pass 0: they sum against a reference taken while staging from
    // each thread's first chunk only (the warp's largest such logit); a warp whose sums
    // come out too large for that (a reference far below a later logit) takes its true
    // maxima and sums again.  At 65536 x 32000 bf16: TVD 94.9 -> 98.5 %, JSD 80.2 -> 81.2 %
    // of the copy bandwidth
    constexpr bool kRef = kTvd || kJsd;
    // TVD, RKL: exponent arguments x c - m c as one fma; JSD: logits clamped to -1e30, (x - m) c
    constexpr bool kFold = !kJsd;
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ __align__(8) uint64_t bar, pbar1, pbar2;
    __shared__ uint32_t s_taddr;
    __shared__ float4 s_slot[kW];  // the warps' values of the exchange in progress
    __shared__ float4 s_res;       // its merged result ...
    __shared__ int s_rerr;         // ... and whether a wait for it gave up

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int csize = p.csize;
    const float c = p.c, inv_tau = p.inv_tau;
    const int rank = (csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    const int cid = blockIdx.x / csize;
    const long long rows = static_cast<long long>(p.G) * p.P;
    const int V = p.V;
    const int e0 = rank * p.span;
    const int n = min(p.span, V - e0);
    const int nv = n / kVec, tail0 = nv * kVec, tail = n - tail0;
    const uint32_t bytes = static_cast<uint32_t>(tail0 * sizeof(In));
    In* zs = reinterpret_cast<In*>(dsm);
    In* ts = zs + p.span;
    float4* recv1 = reinterpret_cast<float4*>(ts + p.span);  // [csize] CTA partials of the first exchange
    float4* recv2 = recv1 + csize;                          // [csize] CTA partials of the second

    // tensor memory for this CTA (the launch keeps resident CTAs x columns <= 512,
    // so the allocation never waits), and the barriers
    if (warp == 0) tm_alloc(&s_taddr, tsh.ncols);
    if (tid == 0) {
        mbar_init(&bar, 1);
        mbar_init(&pbar1, 1);
        mbar_init(&pbar2, 1);
    }
    tm_fence_before_sync();
    if (csize > 1) {  // every CTA's barriers are initialised before any peer pushes to them
        __syncwarp();
        asm volatile("barrier.cluster.arrive.release.aligned;\n"
                     "barrier.cluster.wait.acquire.aligned;" ::: "memory");
    } else {
        __syncthreads();
    }
    tm_fence_after_sync();
    const uint32_t tw = s_taddr + (static_cast<uint32_t>(32 * warp) << 16);

    uint32_t pph = 0;      // pbar1 and pbar2: one phase per row
    bool gave_up = false;  // warp 0: a wait for the peers' partials ran out
    // One exchange: v is this warp's value, merge(x) reduces x over the lanes of
    // warp 0 (lanes past the valid ones hold `ident`) into the same value in
    // every lane, and warp 0 turns the cluster's merge m into the row's values
    // with finish(m, bad) (bad: the row failed); returns them in every thread,
    // `failed` set where a wait gave up or finish found the row bad.
    auto exchange = [&](float4 v, float4 ident, uint64_t* pbar, float4* recv, auto&& merge, auto&& finish,
                        bool& failed) {
        if (lane == 0) s_slot[warp] = v;
        if (warp != 0) {
            named_arrive(1);
            named_sync(2);
            failed = s_rerr != 0;
            return s_res;
        }
        named_sync(1);
        const float4 part = merge(lane < kW ? s_slot[lane] : ident);
        float4 o = ident;
        bool err = false;
        if (csize > 1) {
            if (lane < csize)  // into slot `rank` of CTA `lane`
                st_async_v4(map_rank(&recv[rank], static_cast<uint32_t>(lane)), part,
                            map_rank(pbar, static_cast<uint32_t>(lane)));
            if (lane == 0) mbar_arrive_expect_tx(pbar, static_cast<uint32_t>(csize) * 16u);
            if (!mbar_wait_cluster_bounded(pbar, pph, kTmPartWaitNs)) {
                err = true;
                gave_up = true;
            }
            if (lane < csize) o = recv[lane];
        } else if (lane == 0) {
            o = part;
        }
        bool bad = false;
        const float4 r = finish(merge(o), bad);
        failed = __any_sync(0xffffffffu, err) || bad;
        if (lane == 0) {
            s_res = r;
            s_rerr = failed;
        }
        named_arrive(2);
        return r;
    };

    float nz = 0.f, nt = 0.f;  // the ragged tail entry (tid < tail) of the row in flight ...
    float tz = 0.f, tt = 0.f, tq = 0.f;  // ... and of this row (TVD: tq = q sign(q - p) there)
    // the bulk copies of a row's span (tid 0, when `copy`) and its tail entries
    auto issue = [&](long long row, bool copy) {
        const long long g = row / p.P, pp = row - g * p.P;
        const In* zsrc = static_cast<const In*>(p.draft) + g * p.dsg + pp * p.dsp + e0;
        const In* tsrc = static_cast<const In*>(p.target) + g * p.tsg + pp * p.tsp + e0;
        if (tid == 0 && bytes && copy) {
            fence_proxy_async_smem();  // this CTA's reads of the staging buffer come first
            mbar_arrive_expect_tx(&bar, 2 * bytes);
            bulk_g2s(zs, zsrc, bytes, &bar);
            bulk_g2s(ts, tsrc, bytes, &bar);
        }
        if (tid < tail) {
            nz = Elem<In>::load(zsrc + tail0 + tid);
            nt = Elem<In>::load(tsrc + tail0 + tid);
        }
    };
    // this cluster's run of rows; masked-out rows get loss 0 and are skipped
    long long r0, r1;
    if (cid < tsh.n8) {
        r0 = static_cast<long long>(cid) * tsh.run;
        r1 = min(tsh.end8, r0 + tsh.run);
    } else if (cid < tsh.n8 + tsh.n2) {
        r0 = tsh.end8 + static_cast<long long>(tsh.piece2) * (cid - tsh.n8);
        r1 = min(tsh.end2, r0 + tsh.piece2);
    } else {
        r0 = tsh.end2 + static_cast<long long>(tsh.piece1) * (cid - tsh.n8 - tsh.n2);
        r1 = min(rows, r0 + tsh.piece1);
    }
    auto active = [&](long long r) { return !p.mask || p.mask[r] != 0; };
    if (p.mask && rank == 0 && tid == 0)
        for (long long r = r0; r < r1; ++r)
            if (!p.mask[r]) p.loss[r] = 0.f;
    long long row = r0;
    while (row < r1 && !active(row)) ++row;
    // tid 0: a copy issued and not yet seen landed, and the barrier phase it completes
    bool pending = false;
    uint32_t pend_phase = 0;
    if (row < r1) {
        issue(row, true);
        pending = true;
    }
    auto to_ref = [c](float m, float g) {  // 2^((m - g) c), rounded as the terms are
        if (m == kNegInf) return 0.f;
        return kFold ? ex2(__fmul_rn(m, c) - __fmul_rn(g, c)) : ex2((m - g) * c);
    };
    // the exact part of m c that rn(m c) drops (TVD, RKL: the terms' exponents carry it)
    auto fold_err = [c](float m) { return (kFold && m != kNegInf) ? fmaf(m, c, -__fmul_rn(m, c)) : 0.f; };
    const float beta = p.beta;
    const bool jsd_trivial = kJsd && (beta == 0.f || beta == 1.f);
    uint32_t phase = 0;  // the staging barrier's phase for this row
    bool stop = false;
    for (long long next; row < r1; row = next, phase ^= 1u) {
        next = row + 1;
        while (next < r1 && !active(next)) ++next;
        if (stop) {  // a wait gave up earlier: the rest of this run reports NaN
            if (rank == 0 && tid == 0) p.loss[row] = __int_as_float(0x7fc00000);
            continue;
        }
        // ---- this row's span: shared memory (bounded wait) -> tensor memory; FKL takes
        // pass 0 on the way (this thread's maxima), TVD and JSD the maxima of this
        // thread's first chunk (JSD clamps the logits first, and tensor memory keeps the
        // clamped words)
        const bool landed = !bytes || mbar_wait_bounded(&bar, phase, kStageWaitNs);
        if (tid == 0 && landed) pending = false;
        float mz = kNegInf, mt = kNegInf, tp = kNegInf;
        [[maybe_unused]] uint4 pz = make_uint4(0u, 0u, 0u, 0u), pt = pz;
        [[maybe_unused]] bool piv_tail = false;
        for (int s0 = 0; s0 < tsh.slots; s0 += kTmG) {
            uint4 zr[kTmG], tr[kTmG];
#pragma unroll
            for (int g = 0; g < kTmG; ++g) {
                const int v = tid + kT * (s0 + g);
                zr[g] = (v < nv) ? lds_v4(zs + v * kVec) : make_uint4(0u, 0u, 0u, 0u);
                tr[g] = (v < nv) ? lds_v4(ts + v * kVec) : make_uint4(0u, 0u, 0u, 0u);
                if (kJsd && v < nv) {
                    Elem<In>::clamp_raw(zr[g]);
                    Elem<In>::clamp_raw(tr[g]);
                }
                if ((kStage0 || kRef) && v < nv && (!kRef || (g == 0 && s0 == 0))) {
                    mz = fmaxf(mz, Elem<In>::max_raw(zr[g]));
                    mt = fmaxf(mt, Elem<In>::max_raw(tr[g]));
                }
            }
            tm_st8(tw + 4 * s0, zr[0], zr[1]);
            tm_st8(tw + tsh.t_off + 4 * s0, tr[0], tr[1]);
        }
        tm_wait_st();
        tz = nz;
        tt = nt;
        if ((kStage0 || kRef) && tid < tail) {  // the ragged tail entry, last, as a chunk of one
            if constexpr (kJsd) {
                tz = Elem<In>::clamp1(tz);
                tt = Elem<In>::clamp1(tt);
            }
            mz = fmaxf(mz, tz);
            mt = fmaxf(mt, tt);
        }
        __syncthreads();  // the staging buffer is free
        // ---- the next active row's copy goes in flight while this row is
        // processed; after a copy that gave up (which may still land) none does
        if (next < r1) {
            issue(next, landed);
            if (tid == 0 && landed) {
                pending = true;
                pend_phase = phase ^ 1u;
            }
        }
        const bool werr = __any_sync(0xffffffffu, !landed);

        if constexpr (kRkl) {
            // ---- pass 0 (RKL): this warp's maxima; the raw words of the chunk that first
            // raised this thread's draft maximum, or the tail entry's target logit, are
            // kept and scanned for the pivot once the pass is done
            sweep_tm<In, false, false, true, false, false>(tw, tsh, nv, tail, tz, tt,
                [&](const float*, const float* t, auto tag, int, float cz, float ct, bool, uint4& zr, uint4& tr) {
                    constexpr int kCnt = decltype(tag)::value;
                    if (cz > mz) {
                        mz = cz;
                        if constexpr (kCnt == 1) {
                            piv_tail = true;
                            tp = t[0];
                        } else {
                            piv_tail = false;
                            pz = zr;
                            pt = tr;
                        }
                    }
                    mt = fmaxf(mt, ct);
                });
        }
        if constexpr (kRkl) {
            if (!piv_tail && mz != kNegInf) {  // the first entry of the saved chunk that holds mz
                float z[kVec], t[kVec];
                Elem<In>::unpack(pz, z);
                Elem<In>::unpack(pt, t);
#pragma unroll
                for (int e = kVec - 1; e >= 0; --e)
                    if (z[e] == mz) tp = t[e];
            }
            const float2 pv = warp_max_pivot(mz, tp);
            mz = pv.x;
            tp = pv.y;
        } else {
            mz = warp_max(mz);
        }
        mt = warp_max(mt);

        // the row's maxima (TVD, JSD: its references), and log2 p = (t - gt) c + cu, log2 q = (z - gz) c + cv
        float gz, gt, cu = 0.f, cv;
        float K = 0.f;         // RKL: sum_j q_j ((z_j - gz) - (t_j - tp)) / tau
        int flags = 0;         // RKL: kTmNinf | kTmRklInf over the row
        float sa = 0.f, sb = 0.f;  // TVD: k1, k2 of the gradient; JSD: S = sum q log2(q/m) (in sa)
        bool row_err;
        float loss = 0.f;
        if constexpr (!kMom) {
            // ---- pass 1: sums of 2^((x - m) c) against the warp's reference m (TVD: a
            // warp whose reference is -inf takes m c = 0, and its -inf terms 2^-inf = 0)
            float2 Ez2, Et2;
            auto pass1 = [&]() {
                Ez2 = f2(0.f);
                Et2 = f2(0.f);
                const float Mz = mz == kNegInf ? 0.f : __fmul_rn(mz, c), Mt = mt == kNegInf ? 0.f : __fmul_rn(mt, c);
                sweep_tm<In, false, false, false, false, false>(tw, tsh, nv, tail, tz, tt,
                    [&](const float* z, const float* t, auto tag, int, float, float, bool, uint4& zr, uint4& tr) {
                        constexpr int kCnt = decltype(tag)::value;
                        // JSD's bf16 chunks take x - m straight from the packed words (the
                        // mixed-precision subtract, exact here as the unpacked one is)
                        constexpr bool kRaw = sizeof(In) == 2 && kCnt == 8 && kJsd;
                        const uint32_t zw[4] = {zr.x, zr.y, zr.z, zr.w}, tw4[4] = {tr.x, tr.y, tr.z, tr.w};
                        if constexpr (kCnt == 1) {
                            Ez2.x += kFold ? ex2(fmaf(z[0], c, -Mz)) : ex2((z[0] - mz) * c);
                            Et2.x += kFold ? ex2(fmaf(t[0], c, -Mt)) : ex2((t[0] - mt) * c);
                        } else {
#pragma unroll
                            for (int e = 0; e < kCnt; e += 2) {
                                const float2 zz = make_float2(z[e], z[e + 1]), tt2 = make_float2(t[e], t[e + 1]);
                                float2 a, b;
                                if constexpr (kRaw) {
                                    a = mul2(bf16x2_minus(zw[e / 2], mz), f2(c));
                                    b = mul2(bf16x2_minus(tw4[e / 2], mt), f2(c));
                                } else {
                                    a = kFold ? fma2(zz, f2(c), f2(-Mz)) : mul2(sub2(zz, f2(mz)), f2(c));
                                    b = kFold ? fma2(tt2, f2(c), f2(-Mt)) : mul2(sub2(tt2, f2(mt)), f2(c));
                                }
                                Ez2 = add2(Ez2, make_float2(ex2(a.x), ex2(a.y)));
                                Et2 = add2(Et2, make_float2(ex2(b.x), ex2(b.y)));
                            }
                        }
                    });
            };
            pass1();
            float sz = warp_sum(Ez2.x + Ez2.y), st = warp_sum(Et2.x + Et2.y);
            // a reference from the first chunks keeps every term below 2^32 on the rows this
            // serves; a sum past that (a logit far above the reference), or terms against a
            // -inf reference, send the warp to its true maxima (pass 0) and a second pass 1
            constexpr float kRefMax = 4294967296.f;
            if (__any_sync(0xffffffffu, !(sz < kRefMax) || !(st < kRefMax) || (mz == kNegInf && sz != 0.f) ||
                                            (mt == kNegInf && st != 0.f))) {
                mz = kNegInf;
                mt = kNegInf;
                sweep_tm<In, false, false, true, false, false>(tw, tsh, nv, tail, tz, tt,
                    [&](const float*, const float*, auto, int, float cz, float ct, bool, uint4&, uint4&) {
                        mz = fmaxf(mz, cz);
                        mt = fmaxf(mt, ct);
                    });
                mz = warp_max(mz);
                mt = warp_max(mt);
                pass1();
                sz = warp_sum(Ez2.x + Ez2.y);
                st = warp_sum(Et2.x + Et2.y);
            }
            // ---- exchange 1: the row's references and normalisers (a negative sum flags a failed copy)
            const float4 v1 = make_float4(mz, werr ? -1.f : sz, mt, st);
            bool failed = false;
            const float4 r1v = exchange(v1, make_float4(kNegInf, 0.f, kNegInf, 0.f), &pbar1, recv1,
                [&](float4 x) {
                    const bool e = __any_sync(0xffffffffu, x.y < 0.f);
                    x.y = fmaxf(x.y, 0.f);
                    const float g1 = warp_max(x.x), g2 = warp_max(x.z);
                    const float s1 = warp_sum(x.y * to_ref(x.x, g1)), s2 = warp_sum(x.w * to_ref(x.z, g2));
                    return make_float4(g1, e ? -1.f : s1, g2, s2);
                },
                [&](float4 m, bool& bad) {  // -> (gz, gt, cu, cv)
                    bad = m.y < 0.f;
                    return make_float4(m.x, m.z, -log2_sum(m.w) + fold_err(m.z), -log2_sum(m.y) + fold_err(m.x));
                }, failed);
            row_err = failed;
            gz = r1v.x;
            gt = r1v.y;
            cu = r1v.z;
            cv = r1v.w;
            if (row_err) {  // the row and the rest of the run report NaN
                if (rank == 0 && tid == 0) {
                    p.loss[row] = __int_as_float(0x7fc00000);
                    if (p.status) atomicExch(p.status, static_cast<int32_t>(OSD_ERR_TIMEOUT));
                }
                stop = true;
                continue;
            }
            {
                // ---- pass 2: divergence terms with the global normalisers.  TVD: A = sum
                // |q - p|, S = sum q' with q' = q sign(q - p) (kept in tensor memory in
                // place of the chunk's logits) and Q = sum q; JSD: KL(p||m) and KL(q||m) in bits
                float2 A2 = f2(0.f), B2 = f2(0.f), C2 = f2(0.f);
                if (!jsd_trivial) {
                    sweep_tm<In, false, false, false, false, kTvd, kJsd ? kTmJsdG : kTmG>(tw, tsh, nv, tail, tz, tt,
                        [&](const float* z, const float* t, auto tag, int, float, float, bool, uint4& zr, uint4& tr) {
                            constexpr int kCnt = decltype(tag)::value;
                            constexpr bool kRaw = sizeof(In) == 2 && kCnt == 8;
                            const uint32_t zw[4] = {zr.x, zr.y, zr.z, zr.w}, tw4[4] = {tr.x, tr.y, tr.z, tr.w};
                            [[maybe_unused]] float qs[kCnt];
#pragma unroll
                            for (int e = 0; e < kCnt; e += 2) {
                                const bool two = (e + 1 < kCnt);
                                float2 u, v;
                                if constexpr (kRaw) {
                                    u = fma2(bf16x2_minus(tw4[e / 2], gt), f2(c), f2(cu));
                                    v = fma2(bf16x2_minus(zw[e / 2], gz), f2(c), f2(cv));
                                } else {
                                    u = fma2(sub2(make_float2(t[e], two ? t[e + 1] : t[e]), f2(gt)), f2(c), f2(cu));
                                    v = fma2(sub2(make_float2(z[e], two ? z[e + 1] : z[e]), f2(gz)), f2(c), f2(cv));
                                }
                                const float2 pj = make_float2(ex2(u.x), ex2(u.y)), qj = make_float2(ex2(v.x), ex2(v.y));
                                if constexpr (kJsd) {
                                    // m plus the smallest normal: equal to m above about 2^-102, and
                                    // never 0, so that no lg2 of it is -inf (one FMA, no max)
                                    const float2 m = fma2(pj, f2(beta), fma2(qj, f2(1.f - beta), f2(kMinNormal)));
                                    const float2 lm = make_float2(lg2(m.x), lg2(m.y));
                                    const float2 pw = two ? pj : make_float2(pj.x, 0.f);
                                    const float2 qw = two ? qj : make_float2(qj.x, 0.f);
                                    A2 = fma2(pw, sub2(u, lm), A2);
                                    B2 = fma2(qw, sub2(v, lm), B2);
                                } else {
                                    const float2 df = sub2(qj, pj);
                                    const float2 qq = make_float2(copysignf(qj.x, df.x), copysignf(qj.y, df.y));
                                    qs[e] = qq.x;
                                    if (two) qs[e + 1] = qq.y;
                                    A2.x += fabsf(df.x);
                                    if (two) A2.y += fabsf(df.y);
                                    B2 = add2(B2, two ? qq : make_float2(qq.x, 0.f));
                                    C2 = add2(C2, two ? qj : make_float2(qj.x, 0.f));
                                }
                            }
                            if constexpr (kTvd) {
                                if constexpr (kCnt == 1) tq = qs[0];
                                else pack_q<In>(qs, zr, tr);  // written back to tensor memory by the sweep
                            }
                        });
                }
                // ---- exchange 2: the sums of pass 2
                const float4 v2 = make_float4(warp_sum(A2.x + A2.y), warp_sum(B2.x + B2.y),
                                              kJsd ? 0.f : warp_sum(C2.x + C2.y), 0.f);
                // -> TVD (loss, k1, k2) with the gradient k1 q' + k2 |q'| below; JSD (loss, S)
                const float4 r2v = exchange(v2, make_float4(0.f, 0.f, 0.f, 0.f), &pbar2, recv2,
                    [&](float4 x) {
                        return make_float4(warp_sum(x.x), warp_sum(x.y), kJsd ? 0.f : warp_sum(x.z), 0.f);
                    },
                    [&](float4 m, bool&) {
                        if constexpr (kJsd)
                            return make_float4(jsd_trivial ? 0.f : kLn2 * (beta * m.x + (1.f - beta) * m.y), m.y, 0.f, 0.f);
                        else
                            return make_float4(0.5f * m.x, 0.5f * m.z * inv_tau, -0.5f * m.y * inv_tau, 0.f);
                    }, failed);
                row_err = failed;
                loss = r2v.x;
                sa = r2v.y;
                sb = r2v.z;
            }
        } else {
            // ---- exchange 1: the row's maxima, with RKL's pivot (w flags a failed copy)
            bool failed = false;
            const float4 r1v = exchange(make_float4(mz, tp, mt, werr ? 1.f : 0.f),
                                        make_float4(kNegInf, kNegInf, kNegInf, 0.f), &pbar1, recv1,
                [&](float4 x) {
                    const float2 pv = warp_max_pivot(x.x, x.y);
                    return make_float4(pv.x, pv.y, warp_max(x.z), warp_max(x.w));
                },
                [&](float4 m, bool& bad) {
                    bad = m.w != 0.f;
                    return m;
                }, failed);
            row_err = failed;
            gz = r1v.x;
            gt = r1v.z;
            // the pivot cancels from the loss and the gradient; a -inf one (a -inf target
            // logit at the draft maximum, or no draft mass) becomes 0
            tp = r1v.y == kNegInf ? 0.f : r1v.y;
            if (row_err) {  // the row and the rest of the run report NaN
                if (rank == 0 && tid == 0) {
                    p.loss[row] = __int_as_float(0x7fc00000);
                    if (p.status) atomicExch(p.status, static_cast<int32_t>(OSD_ERR_TIMEOUT));
                }
                stop = true;
                continue;
            }
            {
                // ---- pass 1: the sums and the loss moment against the row's maxima (a row
                // with no mass takes m c = 0): RKL X = sum_j e_z,j ((z_j - gz) - (t_j - tp)),
                // FKL X = sum_j e_t,j (t_j - z_j)
                float2 Ez2 = f2(0.f), Et2 = f2(0.f), X2 = f2(0.f);
                bool ninf = false, rinf = false;
                const float Mz = gz == kNegInf ? 0.f : __fmul_rn(gz, c), Mt = gt == kNegInf ? 0.f : __fmul_rn(gt, c);
                const float2 gz2 = f2(gz), tp2 = f2(tp);
                sweep_tm<In, false, false, false, true, false, kTmMomG>(tw, tsh, nv, tail, tz, tt,
                    [&](const float* z, const float* t, auto tag, int, float, float, bool cninf, uint4&, uint4&) {
                        constexpr int kCnt = decltype(tag)::value;
                        if (kCnt == 1 || cninf) {  // element-wise, with the guards a -inf needs
                            ninf |= cninf;
#pragma unroll
                            for (int e = 0; e < kCnt; ++e) {
                                const float ez = ex2(fmaf(z[e], c, -Mz));
                                const float et = ex2(fmaf(t[e], c, -Mt));
                                Ez2.x += ez;
                                Et2.x += et;
                                if constexpr (kRkl) {
                                    if (z[e] != kNegInf) {
                                        if (t[e] == kNegInf) rinf = true;  // q > 0 = p: the loss is +inf
                                        else X2.x = fmaf(ez, (z[e] - gz) - (t[e] - tp), X2.x);
                                    }
                                } else if (et > 0.f) {  // p > 0 = q makes X, and the loss, +inf
                                    X2.x = fmaf(et, t[e] - z[e], X2.x);
                                }
                            }
                        } else {
#pragma unroll
                            for (int e = 0; e < kCnt; e += 2) {
                                const float2 zz = make_float2(z[e], z[e + 1]), tt2 = make_float2(t[e], t[e + 1]);
                                const float2 a = fma2(zz, f2(c), f2(-Mz)), b = fma2(tt2, f2(c), f2(-Mt));
                                const float2 ez = make_float2(ex2(a.x), ex2(a.y));
                                const float2 et = make_float2(ex2(b.x), ex2(b.y));
                                Ez2 = add2(Ez2, ez);
                                Et2 = add2(Et2, et);
                                if constexpr (kRkl) X2 = fma2(ez, sub2(sub2(zz, gz2), sub2(tt2, tp2)), X2);
                                else X2 = fma2(et, sub2(tt2, zz), X2);
                            }
                        }
                    });
                // ---- exchange 2: the sums, the moment and the flags (OR-ed as bits in w)
                const int wf = warp_or((ninf ? kTmNinf : 0) | (rinf ? kTmRklInf : 0));
                const float4 v2 = make_float4(warp_sum(Ez2.x + Ez2.y), warp_sum(Et2.x + Et2.y),
                                              warp_sum(X2.x + X2.y), __int_as_float(wf));
                // -> (loss, cv, K, flags); FKL (loss, cv, cu, flags)
                const float4 r2v = exchange(v2, make_float4(0.f, 0.f, 0.f, 0.f), &pbar2, recv2,
                    [&](float4 x) {
                        return make_float4(warp_sum(x.x), warp_sum(x.y), warp_sum(x.z),
                                           __int_as_float(warp_or(__float_as_int(x.w))));
                    },
                    [&](float4 m, bool&) {
                        const float Ez = m.x, Et = m.y, X = m.z;
                        const float dz = fold_err(gz), dt = fold_err(gt);
                        const float lr = logf(Ez / Et) - kLn2 * (dz - dt);
                        if constexpr (kFkl)
                            return make_float4((X / Et - (gt - gz)) * inv_tau + lr, -log2_sum(Ez) + dz,
                                               -log2_sum(Et) + dt, m.w);
                        const float l = (__float_as_int(m.w) & kTmRklInf) ? __builtin_huge_valf()
                                                                          : (X / Ez + (gt - tp)) * inv_tau - lr;
                        return make_float4(l, -log2_sum(Ez) + dz, X / Ez * inv_tau, m.w);
                    }, failed);
                row_err = failed;
                loss = r2v.x;
                cv = r2v.y;
                if constexpr (kFkl) cu = r2v.z;
                else K = r2v.z;
                flags = __float_as_int(r2v.w);
            }
        }
        if (rank == 0 && tid == 0) {
            p.loss[row] = row_err ? __int_as_float(0x7fc00000) : loss;
            if (row_err && p.status) atomicExch(p.status, static_cast<int32_t>(OSD_ERR_TIMEOUT));
        }
        if (row_err) {  // the row and the rest of the run report NaN
            stop = true;
            continue;
        }
        pph ^= 1u;

        // ---- pass 3: d loss / d draft logits of the span
        float* orow = p.dlogits + row * V + e0;
        if constexpr (kTvd) {
            // d TVD / d z = q (s Q - S) / (2 tau) with s = sign(q - p), S = sum q s
            // and Q = sum q (1 up to rounding; summed, it cancels S exactly where
            // every s is the same): k1 q' + k2 |q'| with k1 = Q / (2 tau), k2 = -S / (2 tau)
            const float k1 = sa, k2 = sb;
            sweep_tm<In, false, false, false, false, false>(tw, tsh, nv, 0, tz, tt,
                [&](const float*, const float*, auto tag, int j0, float, float, bool, uint4& zr, uint4& tr) {
                    constexpr int kCnt = decltype(tag)::value;
                    if constexpr (kCnt == kVec) {
                        float q[kVec], gr[kVec];
                        unpack_q<In>(zr, tr, q);
#pragma unroll
                        for (int e = 0; e < kVec; ++e) gr[e] = fmaf(k2, fabsf(q[e]), k1 * q[e]);
#pragma unroll
                        for (int e = 0; e < kVec; e += 4) stg_v4(orow + j0 + e, gr[e], gr[e + 1], gr[e + 2], gr[e + 3]);
                    }
                });
            if (tid < tail) orow[tail0 + tid] = fmaf(k2, fabsf(tq), k1 * tq);
        } else {
            // JSD: q (log2(q/m) - S), every probability carrying the gradient's factor,
            // which cancels in log2(q/m); RKL: q ((z - gz) - (t - tp) - X / E) / tau^2,
            // q carrying 1 / tau, and 0 where q = 0 meets an infinite log-ratio; FKL:
            // q - p, both carrying 1 / tau
            const float2 cvs = f2(cv + p.lg_scale), cus = f2(cu + p.lg_scale);
            const bool has_ninf = (flags & kTmNinf) != 0;
            sweep_tm<In, false, false, false, false, false, kJsd ? kTmJsdG : kTmG>(tw, tsh, nv, tail, tz, tt,
                [&](const float* z, const float* t, auto tag, int j0, float, float, bool, uint4& zr, uint4& tr) {
                    constexpr int kCnt = decltype(tag)::value;
                    // RKL's bf16 chunks take x - m from the packed words (mixed-precision subtracts)
                    constexpr bool kRaw = sizeof(In) == 2 && kCnt == 8;
                    const uint32_t zw[4] = {zr.x, zr.y, zr.z, zr.w}, tw4[4] = {tr.x, tr.y, tr.z, tr.w};
                    auto zdiff = [&](int e, float m) {
                        if constexpr (kRaw) return bf16x2_minus(zw[e / 2], m);
                        else return sub2(make_float2(z[e], (e + 1 < kCnt) ? z[e + 1] : z[e]), f2(m));
                    };
                    auto tdiff = [&](int e, float m) {
                        if constexpr (kRaw) return bf16x2_minus(tw4[e / 2], m);
                        else return sub2(make_float2(t[e], (e + 1 < kCnt) ? t[e + 1] : t[e]), f2(m));
                    };
                    float gr[kCnt];
#pragma unroll
                    for (int e = 0; e < kCnt; e += 2) {
                        const bool two = (e + 1 < kCnt);
                        const float2 zd = zdiff(e, gz);
                        const float2 v = fma2(zd, f2(c), cvs);
                        const float2 qj = make_float2(ex2(v.x), ex2(v.y));
                        float2 gg;
                        if constexpr (kRkl) {
                            gg = mul2(qj, fma2(sub2(zd, tdiff(e, tp)), f2(inv_tau), f2(-K)));
                            if (has_ninf) {
                                if (!(qj.x > 0.f)) gg.x = 0.f;
                                if (!(qj.y > 0.f)) gg.y = 0.f;
                            }
                        } else if constexpr (kFkl) {  // (q - p) / tau
                            const float2 u = fma2(tdiff(e, gt), f2(c), cus);
                            gg = sub2(qj, make_float2(ex2(u.x), ex2(u.y)));
                        } else if (jsd_trivial) {
                            gg = f2(0.f);
                        } else {
                            const float2 u = fma2(tdiff(e, gt), f2(c), cus);
                            const float2 pj = make_float2(ex2(u.x), ex2(u.y));
                            const float2 m = fma2(pj, f2(beta), fma2(qj, f2(1.f - beta), f2(kMinNormal)));
                            const float2 lm = make_float2(lg2(m.x), lg2(m.y));
                            gg = mul2(qj, sub2(sub2(v, lm), f2(sa)));
                        }
                        gr[e] = gg.x;
                        if (two) gr[e + 1] = gg.y;
                    }
                    if constexpr (kCnt >= 4) {
#pragma unroll
                        for (int e = 0; e < kCnt; e += 4) stg_v4(orow + j0 + e, gr[e], gr[e + 1], gr[e + 2], gr[e + 3]);
                    } else {
#pragma unroll
                        for (int e = 0; e < kCnt; ++e) orow[j0 + e] = gr[e];
                    }
                });
        }
    }
    if (tid == 0 && pending && bytes) mbar_wait_bounded(&bar, pend_phase, kStageWaitNs);  // a copy still in flight lands first
    if (csize > 1) {
        // every peer has made all its pushes (in the normal course this CTA has
        // received them all); after a wait that gave up, the partial it waited
        // for gets a short while longer to land before the CTA exits
        cluster_arrive_relaxed();
        cluster_wait();
        if (gave_up) {
            mbar_wait_cluster_bounded(&pbar1, pph, 10000000ull);
            mbar_wait_cluster_bounded(&pbar2, pph, 10000000ull);
        }
    }
    tm_fence_before_sync();
    __syncthreads();
    tm_fence_after_sync();
    if (warp == 0) tm_dealloc(s_taddr, tsh.ncols);
}

// ------------------------------------------------------------------ host
// Clusters of more than 8 CTAs need the kernel's non-portable opt-in, set once
// per kernel and device (a function attribute of this process, no device setting).
template <auto kern>
static cudaError_t allow_wide_clusters() {
    static std::atomic<int> done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidValue;
    if (!done[dev].load(std::memory_order_relaxed)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
        done[dev].store(1, std::memory_order_relaxed);
    }
    return cudaSuccess;
}

template <typename In, int kKind, bool kAligned, int kT>
static cudaError_t launch_distill_kind(const DistParams& dp, long long rows, size_t smem, cudaStream_t s) {
    auto kern = distill_kernel<In, kKind, kAligned, kT>;
    if (dp.csize > 8) {
        const cudaError_t e = allow_wide_clusters<distill_kernel<In, kKind, kAligned, kT>>();
        if (e != cudaSuccess) return e;
    }
    if (smem > 48 * 1024) {
        // the opt-in is per device and kernel; set it once, so that later calls
        // (including ones under stream capture) make no attribute call
        static std::atomic<int> allowed[64];
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        if (dev < 0 || dev >= 64 || allowed[dev].load(std::memory_order_relaxed) < static_cast<int>(smem)) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            if (dev >= 0 && dev < 64) {
                int cur = allowed[dev].load(std::memory_order_relaxed);
                while (cur < static_cast<int>(smem) &&
                       !allowed[dev].compare_exchange_weak(cur, static_cast<int>(smem))) {
                }
            }
        }
    }
    return launch(kern, dim3(static_cast<unsigned>(rows * dp.csize)), dim3(kT), smem, s,
                  dp.csize, dp);
}

// Wide CTAs only on the 16-byte path (TVD, whose extra cluster exchange costs
// more with them, always takes kDistThreads).
template <typename In, bool kAligned>
static cudaError_t launch_distill_dtype(osd_loss kind, const DistParams& dp, long long rows, size_t smem,
                                        cudaStream_t s) {
    constexpr int kN = kDistThreads;
    if constexpr (kAligned) {
        constexpr int kWd = kDistThreadsWide;
        if (dp.span >= kDistWideSpan) {
            switch (kind) {
                case OSD_FKL: return launch_distill_kind<In, OSD_FKL, true, kWd>(dp, rows, smem, s);
                case OSD_RKL: return launch_distill_kind<In, OSD_RKL, true, kWd>(dp, rows, smem, s);
                case OSD_JSD: return launch_distill_kind<In, OSD_JSD, true, kWd>(dp, rows, smem, s);
                case OSD_CE: return launch_distill_kind<In, OSD_CE, true, kWd>(dp, rows, smem, s);
                default: break;
            }
        }
    }
    switch (kind) {
        case OSD_FKL: return launch_distill_kind<In, OSD_FKL, kAligned, kN>(dp, rows, smem, s);
        case OSD_RKL: return launch_distill_kind<In, OSD_RKL, kAligned, kN>(dp, rows, smem, s);
        case OSD_JSD: return launch_distill_kind<In, OSD_JSD, kAligned, kN>(dp, rows, smem, s);
        case OSD_CE: return launch_distill_kind<In, OSD_CE, kAligned, kN>(dp, rows, smem, s);
        default: return launch_distill_kind<In, OSD_TVD, kAligned, kN>(dp, rows, smem, s);
    }
}

// The TMEM-staged launch: its shape and the shared-memory request that keeps
// resident CTAs x tensor-memory columns within the SM's 512 columns (so a CTA's
// allocation never waits), looked up once per (device, kernel, span).
struct TmLaunch {
    TmShape shape;
    size_t smem;
    int occ;       // resident CTAs an SM
    int clusters;  // resident clusters of csize CTAs on the GPU
};
// An empty kernel with the TMEM-staged runs' block size and bound on resident
// CTAs.  The cluster occupancy query counts, on it, how many clusters the GPU's
// processing clusters hold at once for a given shared-memory request, which the
// query cannot do on the TMEM kernel itself.  It is never launched.
__global__ void __launch_bounds__(kTmThreads, 7) tm_cluster_probe() {}
template <typename In, int kKind>
static cudaError_t tm_launch_shape(int span, int csize, TmLaunch* out) {
    constexpr int kVec = Elem<In>::kVec;
    const int nv = span / kVec;
    const int slots = (nv + kTmThreads - 1) / kTmThreads;
    const int t_off = 4 * ((slots + kTmG - 1) / kTmG * kTmG);
    uint32_t ncols = 32;
    while (ncols < static_cast<uint32_t>(2 * t_off)) ncols <<= 1;
    if (ncols > 512) return cudaErrorInvalidValue;
    auto kern = distill_tm_kernel<In, kKind>;
    struct Entry {
        int dev, span, csize;
        size_t smem;
        int occ, clusters;
    };
    static std::mutex mu;
    static Entry cache[64];
    static int n_cache = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    {
        std::lock_guard<std::mutex> lock(mu);
        for (int i = 0; i < n_cache; ++i)
            if (cache[i].dev == dev && cache[i].span == span && cache[i].csize == csize) {
                out->shape = TmShape{slots, t_off, ncols, 0, 0, 0, 0, 0, 2, 1};
                out->smem = cache[i].smem;
                out->occ = cache[i].occ;
                out->clusters = cache[i].clusters;
                return cudaSuccess;
            }
    }
    // Every CTA asks for at least ncols x (SM shared memory / 512) bytes of shared
    // memory: then no mix of resident CTAs, of this launch or of concurrent ones
    // with other spans, holds more than the 512 columns, and tcgen05.alloc never
    // has to wait (a CTA waiting for columns while its cluster peers wait for it
    // could otherwise deadlock with another cluster).
    int smem_sm = 0;
    e = cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
    if (e != cudaSuccess) return e;
    const size_t per_col = (size_t(smem_sm) + 511) / 512;
    // the staged span, then the two receive buffers of csize 16-byte partials
    size_t smem = std::max(2 * size_t(span) * sizeof(In) + 2 * size_t(csize) * 16, size_t(ncols) * per_col);
    if (smem > size_t(kDistMaxSmem)) return cudaErrorInvalidValue;
    {
        // the opt-in only ever grows, so that a cached larger launch stays valid
        static int allowed[64] = {};
        std::lock_guard<std::mutex> lock(mu);
        if (dev < 0 || dev >= 64) return cudaErrorInvalidValue;
        if (allowed[dev] < static_cast<int>(smem)) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            allowed[dev] = static_cast<int>(smem);
        }
    }
    // Resident CTAs an SM, from the kernel's limits: the occupancy query reports one
    // CTA an SM for this kernel (it allocates tensor memory) whatever the
    // resources asked for, while ncu shows seven resident at 32 KB spans
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, kern);
    if (e != cudaSuccess) return e;
    int reserved = 0, regs_sm = 0, blocks_sm = 0, threads_sm = 0;
    if ((e = cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&blocks_sm, cudaDevAttrMaxBlocksPerMultiprocessor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&threads_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev)) != cudaSuccess)
        return e;
    const int regs_warp = (fa.numRegs * 32 + 255) / 256 * 256;  // allocated per warp in units of 256
    int occ = std::min(blocks_sm, threads_sm / kTmThreads);
    occ = std::min(occ, static_cast<int>(size_t(smem_sm) / (smem + fa.sharedSizeBytes + size_t(reserved))));
    occ = std::min(occ, regs_sm / (regs_warp * (kTmThreads / 32)));
    occ = std::min(occ, static_cast<int>(512 / ncols));
    if (occ < 1) return cudaErrorInvalidValue;
    // resident clusters: the probe with this launch's shared memory (static included),
    // bounded by the SM count x occ / csize
    int clusters = std::max(1, device_sms() * occ / csize);
    {
        const size_t probe_smem = smem + fa.sharedSizeBytes;
        static int probe_allowed[64] = {};
        static bool probe_wide[64] = {};
        std::lock_guard<std::mutex> lock(mu);
        if (probe_allowed[dev] < static_cast<int>(probe_smem)) {
            e = cudaFuncSetAttribute(tm_cluster_probe, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(probe_smem));
            if (e != cudaSuccess) return e;
            probe_allowed[dev] = static_cast<int>(probe_smem);
        }
        if (csize > 8 && !probe_wide[dev]) {
            e = cudaFuncSetAttribute(tm_cluster_probe, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e != cudaSuccess) return e;
            probe_wide[dev] = true;
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(csize));
        cfg.blockDim = dim3(kTmThreads);
        cfg.dynamicSmemBytes = probe_smem;
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeClusterDimension;
        attr.val.clusterDim.x = static_cast<unsigned>(csize);
        attr.val.clusterDim.y = 1;
        attr.val.clusterDim.z = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        // a failed query leaves the estimate above (the error is not sticky; clear it)
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, tm_cluster_probe, &cfg) == cudaSuccess && n >= 1)
            clusters = std::min(clusters, n);
        else
            (void)cudaGetLastError();
    }
    {
        std::lock_guard<std::mutex> lock(mu);
        if (n_cache < 64) cache[n_cache++] = Entry{dev, span, csize, smem, occ, clusters};
    }
    out->shape = TmShape{slots, t_off, ncols, 0, 0, 0, 0, 0, 2, 1};
    out->smem = smem;
    out->occ = occ;
    out->clusters = clusters;
    return cudaSuccess;
}
template <typename In, int kKind>
static cudaError_t launch_distill_tm(const DistParams& dp, long long rows, cudaStream_t s) {
    if (dp.csize > 8) {
        const cudaError_t e = allow_wide_clusters<distill_tm_kernel<In, kKind>>();
        if (e != cudaSuccess) return e;
    }
    TmLaunch tl;
    const cudaError_t e = tm_launch_shape<In, kKind>(dp.span, dp.csize, &tl);
    if (e != cudaSuccess) return e;
    // Longest runs first: the hardware hands out clusters in about index order, so
    // the last rows, in runs of 2 and then of 1, even out the clusters' finishing
    // times (K = the clusters resident at once: the last K rows singly, the 2K
    // before them in pairs).  With runs of 8 throughout, 6554 rows over about 228
    // resident clusters left some clusters 32 rows and others 24.  The long runs
    // are 8 rows from 16 K rows on, 4 from 8 K, else 2: with few rows per cluster
    // more, shorter runs did better than one wave of long ones (a call of 256 rows
    // of 128256 over the 47 resident 16-CTA clusters: runs of 2, 67.6 us; one wave of
    // runs of 6, 71.7 us), the 16 CTAs of a row waiting on each other twice a row.
    const long long K = tl.clusters;
    TmShape sh = tl.shape;
    sh.run = rows >= 16 * K ? kTmRows : (rows >= 8 * K ? 4 : 2);
    if (dp.mask) {
        // a mask leaves only part of each piece active: runs twice as long and tail
        // pieces of 6 and 3 rows instead of 2 and 1 carry about as much work at 40 %
        // (6554 of 16384 rows of 32128, JSD: 353 against 356 us; runs of 20 and pieces
        // of 5 and 3: 352 us)
        sh.run *= 2;
        sh.piece2 = 6;
        sh.piece1 = 3;
    }
    const long long ones = std::min(rows, K * sh.piece1);
    const long long twos = std::min(rows - ones, 2 * K * sh.piece2);
    sh.end2 = rows - ones;
    sh.end8 = sh.end2 - twos;
    sh.n8 = static_cast<int>((sh.end8 + sh.run - 1) / sh.run);
    sh.n2 = static_cast<int>((twos + sh.piece2 - 1) / sh.piece2);
    const long long n1 = (ones + sh.piece1 - 1) / sh.piece1;
    const long long runs = sh.n8 + sh.n2 + n1;
    return launch(distill_tm_kernel<In, kKind>, dim3(static_cast<unsigned>(runs * dp.csize)),
                  dim3(kTmThreads), tl.smem, s, dp.csize, dp, sh);
}
template <typename In>
static cudaError_t launch_distill_tm_kind(osd_loss kind, const DistParams& dp, long long rows, cudaStream_t s) {
    switch (kind) {
        case OSD_FKL: return launch_distill_tm<In, OSD_FKL>(dp, rows, s);
        case OSD_JSD: return launch_distill_tm<In, OSD_JSD>(dp, rows, s);
        case OSD_RKL: return launch_distill_tm<In, OSD_RKL>(dp, rows, s);
        default: return launch_distill_tm<In, OSD_TVD>(dp, rows, s);
    }
}

// Shared by both entry points: argument checks, shape, and the launch.
static osd_status distill_run(const void* draft_logits, const void* target_logits, osd_dtype dtype, int G,
                              int P, int V, int64_t d_stride_g, int64_t d_stride_p, int64_t t_stride_g,
                              int64_t t_stride_p, const uint8_t* mask, const int32_t* accepted, int k,
                              int32_t* seq_of_row, int32_t* count, osd_loss kind, float beta,
                              float temperature, float* loss, float* dlogits, int32_t* status, void* stream) {
    if (dtype != OSD_F32 && dtype != OSD_BF16) return OSD_ERR_INVALID_ARG;
    if (kind < OSD_FKL || kind > OSD_CE) return OSD_ERR_INVALID_ARG;
    if (!(temperature > 0.f) || !std::isfinite(temperature)) return OSD_ERR_INVALID_ARG;
    if (G < 0 || P < 0 || V < 1) return OSD_ERR_INVALID_ARG;
    if (d_stride_g < 0 || d_stride_p < 0 || t_stride_g < 0 || t_stride_p < 0) return OSD_ERR_INVALID_ARG;
    if (kind == OSD_JSD && !(beta >= 0.f && beta <= 1.f)) return OSD_ERR_INVALID_ARG;
    const size_t es = dtype_size(dtype);
    // rows on 16-byte boundaries take the vectorised path (bulk copies, 16-byte stores)
    auto row_ok = [&](int64_t stride, int n) { return n <= 1 || (stride * int64_t(es)) % 16 == 0; };
    const int p_rows = accepted ? k : P;  // the position index runs over k rows in accepted mode
    const bool aligned = aligned_to(draft_logits, 16) && aligned_to(target_logits, 16) &&
                         aligned_to(dlogits, 16) && (size_t(V) * 4) % 16 == 0 &&
                         row_ok(d_stride_g, G) && row_ok(d_stride_p, p_rows) && row_ok(t_stride_g, G) &&
                         row_ok(t_stride_p, p_rows);
    // the TMEM-staged runs (if the span fits) for TVD, JSD, RKL and FKL, where they
    // measured faster: TVD 95.1 % against 70.1 % of the HBM peak, JSD 71.9 % against
    // 63.0 %, RKL 95.5 % against 86.4 %, FKL 100.6 % against 90.9 % of the measured
    // copy bandwidth (65536 x 32000 bf16); CE stays at 96.3 % on the per-row kernel.
    // Rows chosen by verification stay on the per-row kernel: on the runs, 32 rows
    // of 32000 took 12.8 against 10.4 us, and 256 of 128256 no less time
    const bool tm_path = aligned && !accepted &&
                         (kind == OSD_TVD || kind == OSD_JSD || kind == OSD_RKL || kind == OSD_FKL);
    int csize = 1, span = V;
    // JSD, with the most work per entry, stages best in longer spans on the per-row
    // kernel; the TMEM-staged runs take the 32 KB spans for every kind.  (At
    // V = 32000 a span of 8000 bf16 entries leaves room for seven CTAs an SM; spans
    // cut in 16-byte steps to seven CTAs at V = 32128, five CTAs a row instead of
    // four, measured 8 % slower for JSD than four spans of 8064 at six CTAs.)
    size_t span_bytes = (kind == OSD_JSD && !tm_path) ? kDistSpanBytesJsd : kDistSpanBytes;
    // no more rows than SMs: half-length spans put twice the CTAs to work on them
    // (measured 6-12 % less latency at 4 and 128 rows of 32000)
    if (static_cast<long long>(G) * P <= device_sms()) span_bytes /= 2;
    if (!row_span_shape(V, es, span_bytes, kDistMaxCluster, kDistMaxSmem, &csize, &span))
        return OSD_ERR_UNSUPPORTED;
    // on the TMEM-staged runs, rows that need more than 8 spans of the target size
    // take up to 16 CTAs: spans that fit 64 columns of tensor memory and six CTAs
    // an SM instead of 128 columns and two (2048 x 128256 bf16: FKL 77.7 against
    // 75.6 %, RKL 71.5 against 67.9 %, TVD 71.8 against 65.0 %, JSD 55.3 against
    // 54.3 %); the per-row kernel keeps at most 8 (measured no faster)
    if (tm_path && csize == kDistMaxCluster && size_t(span) * 2 * es > span_bytes &&
        !row_span_shape(V, es, span_bytes, kDistMaxClusterWide, kDistMaxSmem, &csize, &span))
        return OSD_ERR_UNSUPPORTED;
    const long long rows = static_cast<long long>(G) * P;
    if (rows * csize > INT_MAX) return OSD_ERR_UNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (status && !aligned_to(status, 4)) return OSD_ERR_INVALID_ARG;
    if ((seq_of_row && !aligned_to(seq_of_row, 4)) || (count && !aligned_to(count, 4))) return OSD_ERR_INVALID_ARG;
    if (rows == 0) {
        if (status) {
            const cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
            if (e != cudaSuccess) return OSD_ERR_CUDA;
        }
        return count ? from_cuda(cudaMemsetAsync(count, 0, sizeof(int32_t), s)) : OSD_OK;
    }
    if (!draft_logits || !target_logits || !loss || !dlogits) return OSD_ERR_INVALID_ARG;
    if (!aligned_to(draft_logits, es) || !aligned_to(target_logits, es) || !aligned_to(loss, 4) ||
        !aligned_to(dlogits, 4))
        return OSD_ERR_INVALID_ARG;
    if (status) {
        const cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
        if (e != cudaSuccess) return OSD_ERR_CUDA;
    }
    DistParams dp;
    dp.draft = draft_logits; dp.target = target_logits;
    dp.G = G; dp.P = P; dp.V = V;
    dp.dsg = d_stride_g; dp.dsp = d_stride_p; dp.tsg = t_stride_g; dp.tsp = t_stride_p;
    dp.mask = mask; dp.beta = beta; dp.loss = loss; dp.dlogits = dlogits; dp.status = status;
    dp.accepted = accepted; dp.k = k; dp.seq_of_row = seq_of_row; dp.count = count;
    dp.c = static_cast<float>(1.4426950408889634074 / static_cast<double>(temperature));
    dp.inv_tau = static_cast<float>(1.0 / static_cast<double>(temperature));
    {
        double scale = 1.0 / static_cast<double>(temperature);
        if (kind == OSD_JSD) scale *= (1.0 - static_cast<double>(beta)) * 0.69314718055994530942;
        dp.lg_scale = scale > 0.0 ? static_cast<float>(std::log2(scale)) : 0.f;  // beta = 1: gradient is 0
    }
    dp.csize = csize; dp.span = span;
    const size_t smem = 2 * size_t(span) * es;
    cudaError_t e;
    // 16-byte rows and a span that fits tensor memory: the TMEM-staged runs
    const bool tm = tm_path && span / static_cast<int>(16 / es) <= kTmMaxChunks;
    if (tm) {
        e = (dtype == OSD_BF16) ? launch_distill_tm_kind<__nv_bfloat16>(kind, dp, rows, s)
                                : launch_distill_tm_kind<float>(kind, dp, rows, s);
        return from_cuda(e);
    }
    if (dtype == OSD_BF16)
        e = aligned ? launch_distill_dtype<__nv_bfloat16, true>(kind, dp, rows, smem, s)
                    : launch_distill_dtype<__nv_bfloat16, false>(kind, dp, rows, smem, s);
    else
        e = aligned ? launch_distill_dtype<float, true>(kind, dp, rows, smem, s)
                    : launch_distill_dtype<float, false>(kind, dp, rows, smem, s);
    return from_cuda(e);
}

}  // namespace osd

extern "C" osd_status osd_distill(const void* draft_logits, const void* target_logits, osd_dtype dtype,
                                  int G, int P, int V, int64_t d_stride_g, int64_t d_stride_p,
                                  int64_t t_stride_g, int64_t t_stride_p, const uint8_t* mask, osd_loss kind,
                                  float beta, float temperature, float* loss, float* dlogits, int32_t* status,
                                  void* stream) {
    return osd::distill_run(draft_logits, target_logits, dtype, G, P, V, d_stride_g, d_stride_p, t_stride_g,
                            t_stride_p, mask, nullptr, 0, nullptr, nullptr, kind, beta, temperature, loss,
                            dlogits, status, stream);
}

extern "C" osd_status osd_distill_accepted(const void* draft_logits, const void* target_logits,
                                           osd_dtype dtype, int B, int k, int V, const int32_t* accepted,
                                           osd_loss kind, float beta, float temperature, float* loss,
                                           float* dlogits, int32_t* seq_of_row, int32_t* count,
                                           int32_t* status, void* stream) {
    if (k < 1 || B < 0 || V < 1) return OSD_ERR_INVALID_ARG;
    if (B > 0 && (!accepted || !osd::aligned_to(accepted, 4))) return OSD_ERR_INVALID_ARG;
    const int64_t kv = int64_t(k) * V;
    return osd::distill_run(draft_logits, target_logits, dtype, B, 1, V, kv, V, kv + V, V, nullptr,
                            B > 0 ? accepted : nullptr, k, seq_of_row, count, kind, beta, temperature, loss,
                            dlogits, status, stream);
}
