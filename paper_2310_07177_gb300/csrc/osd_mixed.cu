// osd_mixed.cu -- mixed-token sampling (Section 4.1 of the paper): one draw
// per position from beta p + (1 - beta) q_theta, p = softmax(t / tau),
// q = softmax(z / tau), by inverse CDF in ascending vocabulary order,
// j* = min{ j : C_j > u W } (the convention of the verifier's extra token).
//
// One thread-block cluster per row; each CTA stages its span of both rows in
// shared memory (osd_rowspan.cuh) and reads HBM once:
//
//   pass 0  block maxima of both rows;
//   pass 1  sums of 2^((x - m) c) of both rows over each warp's range, a
//           contiguous quarter of the span: the pieces of the CDF;
//   merge   warp 0 of every CTA gathers the cluster's CTA sums over DSMEM,
//           forms both normalisers and the mixture mass of every CTA, and finds
//           by an fp64 scan in rank order the CTA that holds u W;
//   pick    warp 0 of that CTA takes the range that holds u W from the range
//           sums and rescans it in steps of 32 chunks with fp64 prefix sums.
//
// Every entry is exponentiated once, plus once more for the one range that is
// rescanned: two ex2 per entry for both rows together.  At the HBM rate that
// is about three quarters of the SM's ex2 throughput, which with the
// per-row merge sets this kernel's speed.
#include <atomic>
#include <climits>
#include <cmath>
#include <cstdint>

#include "osd.h"
#include "osd_device.cuh"
#include "osd_host.hpp"
#include "osd_rowspan.cuh"

namespace osd {

constexpr int kMixMaxCluster = 8;
constexpr int kMixSpanBytes = 32768;     // target bytes of both rows per CTA
constexpr int kMixMaxSmem = 192 * 1024;  // largest staging buffer per CTA
constexpr int kGroups = 8;               // CDF pieces per warp range (kRowWarps * kGroups = 32)
static_assert(kRowWarps * kGroups == 32, "one CDF piece per lane of the picking warp");

struct MixParams {
    const void* draft;
    const void* target;
    int V;
    long long dstride, tstride;  // elements between consecutive rows
    const float* uniforms;
    float beta;
    float c_hi, c_lo;  // log2(e) / tau as a float pair (c_lo > 0)
    int32_t* tokens;
    float* cdf_gap;
    int32_t* status;
    int csize;  // CTAs per row (cluster size)
    int span;   // vocabulary entries per CTA
};

// One CTA's partial: block maxima and the sums of both rows against them.
struct MixStats {
    float mz, Z, mt, T;
    int err;
};

template <typename In, bool kAligned>
__global__ void __launch_bounds__(kRowThreads) mixed_sample_kernel(MixParams p) {
    using E = Elem<In>;
    constexpr int kVec = kAligned ? E::kVec : 1;  // entries per chunk
    extern __shared__ __align__(128) unsigned char dsm[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ int s_err;
    __shared__ float2 red_m[kRowWarps];
    __shared__ float2 s_rng[kRowWarps];  // (sum 2^((t-m)c), sum 2^((z-m)c)) of each warp's range
    __shared__ float2 s_piece[kRowWarps * kGroups];  // the same over each run of steps
    __shared__ MixStats s_mine;
    __shared__ int s_owner, s_mode, s_bad;
    __shared__ float s_a, s_b;
    __shared__ double s_tau, s_W, s_base;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int csize = p.csize;
    const int rank = (csize > 1) ? static_cast<int>(cluster_rank()) : 0;
    const long long row = blockIdx.x / csize;
    const In* zrow = static_cast<const In*>(p.draft) + row * p.dstride;
    const In* trow = static_cast<const In*>(p.target) + row * p.tstride;
    const int V = p.V;
    const int e0 = rank * p.span;
    const int n = min(p.span, V - e0);
    In* zs = reinterpret_cast<In*>(dsm);
    In* ts = zs + p.span;
    const int err_local = stage_span<In, kAligned>(zs, ts, zrow + e0, trow + e0, n, &bar, &s_err);
    const float ch = p.c_hi, cl = p.c_lo;

    // ---- pass 0: block maxima
    float mz = kNegInf, mt = kNegInf;
    if (!err_local) {
        sweep<In, kAligned, false, false, true>(zs, ts, n, [&](const float*, const float*, auto, int, float cz,
                                                               float ct, bool, const uint4&, const uint4&) {
            mz = fmaxf(mz, cz);
            mt = fmaxf(mt, ct);
        });
    }
    const float2 bm = block_max2<false>(mz, mt, red_m);  // red_m has no readers yet
    const float gzb = bm.x, gtb = bm.y;
    const bool zok = gzb != kNegInf, tok = gtb != kNegInf;  // a span of -inf has no mass

    // chunk at entry j (kVec entries; past `end` they read as -inf)
    auto load_chunk = [&](int j, int end, float* z, float* t) {
        if (kAligned && j + kVec <= end) {
            E::unpack(lds_v4(zs + j), z);
            E::unpack(lds_v4(ts + j), t);
        } else {
#pragma unroll
            for (int e = 0; e < kVec; ++e) {
                z[e] = (j + e < end) ? E::lds(zs + j + e) : kNegInf;
                t[e] = (j + e < end) ? E::lds(ts + j + e) : kNegInf;
            }
        }
    };
    // 2^((x - m) c) of a pair, the exponent from the exact difference times c_hi + c_lo
    auto exp_pair = [&](float x0, float x1, float m) {
        const float2 d = sub2(make_float2(x0, x1), f2(m));
        const float2 g = fma2(d, f2(ch), mul2(d, f2(cl)));
        return make_float2(ex2(g.x), ex2(g.y));
    };
    auto exp_one = [&](float x, float m) { return ex2(mul_c(x - m, ch, cl)); };

    // ---- pass 1: each warp's contiguous range [lo(w), lo(w + 1)) in steps of 32 chunks,
    // the steps split into kGroups runs whose sums stay in registers until the loop ends:
    // kRowWarps x kGroups pieces of the CDF, with no shuffle inside the loop
    const int nchunks = (n + kVec - 1) / kVec;
    const int range_len = (nchunks + kRowWarps - 1) / kRowWarps * kVec;
    auto range_lo = [&](int w) { return min(n, w * range_len); };
    const int steps = (range_len / kVec + 31) / 32;      // per warp
    const int per_group = (steps + kGroups - 1) / kGroups;
    // a span with no mass: its logits are -inf, and so are x - 0
    const float gz_ref = zok ? gzb : 0.f, gt_ref = tok ? gtb : 0.f;
    {
        const int lo_w = range_lo(warp), hi_w = range_lo(warp + 1);
        float Tg[kGroups], Zg[kGroups];
#pragma unroll
        for (int g = 0; g < kGroups; ++g) {
            float2 T2 = f2(0.f), Z2 = f2(0.f);
            if (!err_local) {
                const int s_end = min((g + 1) * per_group, steps);
                for (int st = g * per_group; st < s_end; ++st) {
                    const int j = lo_w + (st * 32 + lane) * kVec;
                    if (j < hi_w) {
                        float z[kVec], t[kVec];
                        load_chunk(j, hi_w, z, t);
                        if constexpr (kVec == 1) {
                            T2.x += exp_one(t[0], gt_ref);
                            Z2.x += exp_one(z[0], gz_ref);
                        } else {
#pragma unroll
                            for (int e = 0; e < kVec; e += 2) {
                                T2 = add2(T2, exp_pair(t[e], t[e + 1], gt_ref));
                                Z2 = add2(Z2, exp_pair(z[e], z[e + 1], gz_ref));
                            }
                        }
                    }
                }
            }
            Tg[g] = T2.x + T2.y;
            Zg[g] = Z2.x + Z2.y;
        }
        for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
            for (int g = 0; g < kGroups; ++g) {
                Tg[g] += __shfl_xor_sync(0xffffffffu, Tg[g], o);
                Zg[g] += __shfl_xor_sync(0xffffffffu, Zg[g], o);
            }
        }
        if (lane == 0) {
            float Tw = 0.f, Zw = 0.f;
#pragma unroll
            for (int g = 0; g < kGroups; ++g) {
                s_piece[warp * kGroups + g] = make_float2(Tg[g], Zg[g]);
                Tw += Tg[g];
                Zw += Zg[g];
            }
            s_rng[warp] = make_float2(Tw, Zw);
        }
    }
    __syncthreads();
    if (tid == 0) {
        float T = 0.f, Z = 0.f;
#pragma unroll
        for (int w = 0; w < kRowWarps; ++w) {
            T += s_rng[w].x;
            Z += s_rng[w].y;
        }
        s_mine = MixStats{gzb, Z, gtb, T, err_local};
    }
    if (csize > 1) cluster_sync_publish(tid == 0); else __syncthreads();

    // ---- merge: every CTA's warp 0 derives the same normalisers, masses and owner
    if (warp == 0) {
        MixStats o{kNegInf, 0.f, kNegInf, 0.f, 0};
        if (lane < csize) {
            if (lane == rank) {
                o = s_mine;
            } else {
                const uint32_t base = map_rank(&s_mine, lane);
                o.mz = ld_dsmem_f32(base + offsetof(MixStats, mz));
                o.Z = ld_dsmem_f32(base + offsetof(MixStats, Z));
                o.mt = ld_dsmem_f32(base + offsetof(MixStats, mt));
                o.T = ld_dsmem_f32(base + offsetof(MixStats, T));
                o.err = ld_dsmem_s32(base + offsetof(MixStats, err));
            }
        }
        float gz = o.mz, gt = o.mt;
        int err = o.err;
        for (int off = 16; off > 0; off >>= 1) {
            gz = fmaxf(gz, __shfl_xor_sync(0xffffffffu, gz, off));
            gt = fmaxf(gt, __shfl_xor_sync(0xffffffffu, gt, off));
            err |= __shfl_xor_sync(0xffffffffu, err, off);
        }
        const float sz = (o.mz == kNegInf) ? 0.f : exp_one(o.mz, gz);
        const float st = (o.mt == kNegInf) ? 0.f : exp_one(o.mt, gt);
        float Ez = o.Z * sz, Et = o.T * st;
        for (int off = 16; off > 0; off >>= 1) {
            Ez += __shfl_xor_sync(0xffffffffu, Ez, off);
            Et += __shfl_xor_sync(0xffffffffu, Et, off);
        }
        // CTA `lane`'s weights: w_j = a 2^((t_j - m_t)c) + b 2^((z_j - m_z)c) against its block maxima
        const float a = (Et > 0.f) ? p.beta * st / Et : 0.f;
        const float b = (Ez > 0.f) ? (1.f - p.beta) * sz / Ez : 0.f;
        const double mass = double(a) * double(o.T) + double(b) * double(o.Z);
        const double incl = warp_incl_scan_f64(mass);
        const double W = __shfl_sync(0xffffffffu, incl, 31);
        const double tau = double(p.uniforms[row]) * W;
        int mode = 0, owner;  // mode 0: inverse CDF; 1: the largest j with w_j > 0
        double base = 0.0;
        const unsigned hit = __ballot_sync(0xffffffffu, lane < csize && incl > tau);
        if (hit) {
            owner = __ffs(hit) - 1;
            base = __shfl_sync(0xffffffffu, incl - mass, owner);
        } else {
            mode = 1;
            const unsigned pos = __ballot_sync(0xffffffffu, lane < csize && mass > 0.0);
            owner = pos ? 31 - __clz(pos) : 0;
        }
        if (lane == rank) {
            s_a = a;
            s_b = b;
        }
        if (lane == 0) {
            s_owner = owner;
            s_mode = mode;
            s_tau = tau;
            s_W = W;
            s_base = base;
            s_bad = err;
        }
    }
    __syncthreads();
    if (csize > 1) cluster_arrive_relaxed();  // finished reading the other CTAs' shared memory

    if (s_bad) {
        if (rank == 0 && tid == 0) {
            p.tokens[row] = -1;
            if (p.cdf_gap) p.cdf_gap[row] = __int_as_float(0x7fc00000);
            if (p.status) atomicExch(p.status, static_cast<int32_t>(OSD_ERR_TIMEOUT));
        }
    } else if (rank == s_owner && warp == 0) {
        // ---- pick: the piece (lane l holds piece l, in vocabulary order), then the entry, in fp64
        const float a = s_a, b = s_b;
        const double tau = s_tau, W = s_W;
        int mode = s_mode;
        const double mass = double(a) * double(s_piece[lane].x) + double(b) * double(s_piece[lane].y);
        const double incl = s_base + warp_incl_scan_f64(mass);
        int piece = -1;
        double run = 0.0;
        if (mode == 0) {
            const unsigned h = __ballot_sync(0xffffffffu, incl - mass <= tau && incl > tau);
            if (h) {
                piece = __ffs(h) - 1;
                run = __shfl_sync(0xffffffffu, incl - mass, piece);
            } else {
                mode = 1;
            }
        }
        if (mode == 1) {  // the last piece with positive mass
            const unsigned pos = __ballot_sync(0xffffffffu, mass > 0.0);
            piece = pos ? 31 - __clz(pos) : 0;
        }
        const int pw = piece / kGroups, pg = piece % kGroups;
        const int lo = range_lo(pw), hi = range_lo(pw + 1);
        const int s_end = min((pg + 1) * per_group, steps);
        int pick = -1, last_pos = -1;
        double gap = 0.0;
        bool found = false;
        for (int st = pg * per_group; st < s_end; ++st) {  // warp-uniform trip count
            const int j = lo + (st * 32 + lane) * kVec;
            float z[kVec], t[kVec], w[kVec];
            load_chunk(j, hi, z, t);  // past the range end the entries read as -inf: weight 0
#pragma unroll
            for (int e = 0; e < kVec; ++e) {
                const float pt = exp_one(t[e], gt_ref);
                const float qz = exp_one(z[e], gz_ref);
                w[e] = fmaf(a, pt, b * qz);
                if (w[e] > 0.f) last_pos = j + e;
            }
            double mine = 0.0;
#pragma unroll
            for (int e = 0; e < kVec; ++e) mine += double(w[e]);
            const double wincl = warp_incl_scan_f64(mine);
            if (mode == 0) {
                const double excl = run + wincl - mine;
                const unsigned h = __ballot_sync(0xffffffffu, excl <= tau && excl + mine > tau);
                if (h) {
                    if (lane == __ffs(h) - 1) {
                        double C = excl;
                        for (int e = 0; e < kVec; ++e) {
                            const double Cprev = C;
                            C += double(w[e]);
                            if (C > tau) {
                                pick = j + e;
                                gap = fmin(C - tau, tau - Cprev) / W;
                                break;
                            }
                        }
                        if (pick < 0) {  // the lane's entries pass tau only after rounding
                            pick = last_pos;
                            gap = 0.0;
                        }
                    }
                    found = true;
                }
            }
            if (found) break;
            run += __shfl_sync(0xffffffffu, wincl, 31);
        }
        if (!found) {  // mode 1, or rounding left tau past the piece: the largest j with w_j > 0
            int lp = last_pos;
            for (int off = 16; off > 0; off >>= 1) lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, off));
            if (lane == 0) {
                pick = (lp >= 0) ? lp : lo;
                gap = (mode == 1) ? (W - tau) / W : 0.0;
            }
        }
        if (pick >= 0) {
            p.tokens[row] = e0 + pick;
            if (p.cdf_gap) p.cdf_gap[row] = float(gap);
        }
    }
    if (csize > 1) cluster_wait();  // keep this CTA's partial readable until every peer is done
}

template <typename In, bool kAligned>
static cudaError_t launch_mixed(const MixParams& mp, int N, size_t smem, cudaStream_t s) {
    auto kern = mixed_sample_kernel<In, kAligned>;
    if (smem > 48 * 1024) {
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
    return launch(kern, dim3(static_cast<unsigned>(static_cast<long long>(N) * mp.csize)), dim3(kRowThreads), smem, s,
                  mp.csize, mp);
}

}  // namespace osd

extern "C" osd_status osd_mixed_sample(const void* draft_logits, const void* target_logits, osd_dtype dtype, int N,
                                       int V, int64_t d_stride, int64_t t_stride, const float* uniforms, float beta,
                                       float temperature, int32_t* tokens, float* cdf_gap, int32_t* status,
                                       void* stream) {
    using namespace osd;
    if (dtype != OSD_F32 && dtype != OSD_BF16) return OSD_ERR_INVALID_ARG;
    if (N < 0 || V < 1 || d_stride < 0 || t_stride < 0) return OSD_ERR_INVALID_ARG;
    if (!(beta >= 0.f && beta <= 1.f)) return OSD_ERR_INVALID_ARG;
    if (!(temperature > 0.f) || !std::isfinite(temperature)) return OSD_ERR_INVALID_ARG;
    const size_t es = dtype_size(dtype);
    int csize = 1, span = V;
    if (!row_span_shape(V, es, kMixSpanBytes, kMixMaxCluster, kMixMaxSmem, &csize, &span))
        return OSD_ERR_UNSUPPORTED;
    if (static_cast<long long>(N) * csize > INT_MAX) return OSD_ERR_UNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (status && !aligned_to(status, 4)) return OSD_ERR_INVALID_ARG;
    if (status) {
        const cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
        if (e != cudaSuccess) return OSD_ERR_CUDA;
    }
    if (N == 0) return OSD_OK;
    if (!draft_logits || !target_logits || !uniforms || !tokens) return OSD_ERR_INVALID_ARG;
    if (!aligned_to(draft_logits, es) || !aligned_to(target_logits, es) || !aligned_to(uniforms, 4) ||
        !aligned_to(tokens, 4) || (cdf_gap && !aligned_to(cdf_gap, 4)))
        return OSD_ERR_INVALID_ARG;
    auto row_ok = [&](int64_t stride) { return N <= 1 || (stride * int64_t(es)) % 16 == 0; };
    const bool aligned = aligned_to(draft_logits, 16) && aligned_to(target_logits, 16) && row_ok(d_stride) &&
                         row_ok(t_stride);
    MixParams mp;
    mp.draft = draft_logits;
    mp.target = target_logits;
    mp.V = V;
    mp.dstride = d_stride;
    mp.tstride = t_stride;
    mp.uniforms = uniforms;
    mp.beta = beta;
    split_scale(temperature, &mp.c_hi, &mp.c_lo);
    mp.tokens = tokens;
    mp.cdf_gap = cdf_gap;
    mp.status = status;
    mp.csize = csize;
    mp.span = span;
    const size_t smem = 2 * size_t(span) * es;
    cudaError_t e;
    if (dtype == OSD_BF16)
        e = aligned ? launch_mixed<__nv_bfloat16, true>(mp, N, smem, s) : launch_mixed<__nv_bfloat16, false>(mp, N, smem, s);
    else
        e = aligned ? launch_mixed<float, true>(mp, N, smem, s) : launch_mixed<float, false>(mp, N, smem, s);
    return from_cuda(e);
}
